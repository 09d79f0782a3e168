// Tree-masked attention over the paged KV cache (tree verification, prefill chunks
// and the draft's full-context layer).
//
// Keys of sequence b: the n_ctx[b] committed rows (visible to every query) followed by
// n_local rows at slots n_ctx..n_ctx+n_local-1; query i sees local row j iff bit j of
// anc[q_local0 + i] is set (a tree node's ancestors-or-self, or a causal chain).
// KV layout: pool[layer][block][head][plane][16 rows][hd], page_table[b][slot / 16];
// planes K, V (fp32 models, plain bf16) or K_hi, K_lo, V_hi, V_lo (bf16 two-term split).
//
// Grid (splits, heads, batch).  Each CTA loads every KV tile of its key range once
// into shared memory for all the sequence's queries; online softmax in fp32.  This
// file holds the SIMT kernel (fp32 models, and bf16 models with head_dim 64), whose
// splits merge in the last CTA of each (b, h) through a global workspace, and the
// dispatch; bf16 models with head_dim 128 take the tensor-core kernel of
// attention_tc.cu, which can also fuse RoPE and the KV write of the step's fresh rows.
#include <algorithm>
#include <cmath>

#include <mutex>

#include "common.cuh"
#include "launch.cuh"
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


constexpr int MAX_SPLITS = 16;

// Merge the per-split partials (unnormalised output, running max, running sum) of the
// nq queries of one (b, h), in split order.  Run by the last CTA of the pair; every
// thread takes part: first the per-query weights exp(m_s - M) / L into shared memory,
// then the outputs, 4 dims per item, up to 8 items x 4 splits of loads in flight.
template <typename T>
__device__ void combine_splits(const AttnParams& p, const float* wsb, int nq, int hd, int b, int h, T* out,
                               T* out_lo, float* s_w /* [nq][MAX_SPLITS] */) {
  const size_t rec = hd + 4;
  for (int qi = threadIdx.x; qi < nq; qi += blockDim.x) {
    float mv[MAX_SPLITS], lv[MAX_SPLITS];
#pragma unroll
    for (int sp = 0; sp < MAX_SPLITS; ++sp) {
      mv[sp] = -INFINITY;
      lv[sp] = 0.f;
      if (sp < p.splits) {
        const float* w = wsb + (static_cast<size_t>(sp) * p.nq_max + qi) * rec + hd;
        mv[sp] = __ldcg(w);
        lv[sp] = __ldcg(w + 1);
      }
    }
    float M = -INFINITY;
#pragma unroll
    for (int sp = 0; sp < MAX_SPLITS; ++sp) M = fmaxf(M, mv[sp]);
    float L = 0.f;
#pragma unroll
    for (int sp = 0; sp < MAX_SPLITS; ++sp) {
      mv[sp] = (M == -INFINITY || mv[sp] == -INFINITY) ? 0.f : expf(mv[sp] - M);
      L += mv[sp] * lv[sp];
    }
    const float inv = L > 0.f ? 1.f / L : 0.f;
#pragma unroll
    for (int sp = 0; sp < MAX_SPLITS; ++sp)
      if (sp < p.splits) s_w[qi * MAX_SPLITS + sp] = mv[sp] * inv;
  }
  __syncthreads();
  constexpr int J = 8;
  const int c4n = hd / 4;
  const int items = nq * c4n;
  const int nt = blockDim.x;
  for (int it0 = threadIdx.x; it0 < items; it0 += J * nt) {
    float4 acc[J];
#pragma unroll
    for (int j = 0; j < J; ++j) acc[j] = make_float4(0.f, 0.f, 0.f, 0.f);
    for (int sp0 = 0; sp0 < p.splits; sp0 += 4) {
      float4 v[J][4];
#pragma unroll
      for (int j = 0; j < J; ++j) {
        const int it = it0 + j * nt;
        const int qi = it / c4n, c = (it % c4n) * 4;
#pragma unroll
        for (int u = 0; u < 4; ++u)
          if (it < items && sp0 + u < p.splits)
            v[j][u] = __ldcg(reinterpret_cast<const float4*>(wsb + (static_cast<size_t>(sp0 + u) * p.nq_max + qi) * rec + c));
      }
#pragma unroll
      for (int j = 0; j < J; ++j) {
        const int it = it0 + j * nt;
        if (it >= items) continue;
        const int qi = it / c4n;
#pragma unroll
        for (int u = 0; u < 4; ++u)
          if (sp0 + u < p.splits) {
            const float e = s_w[qi * MAX_SPLITS + sp0 + u];
            acc[j].x += e * v[j][u].x; acc[j].y += e * v[j][u].y; acc[j].z += e * v[j][u].z; acc[j].w += e * v[j][u].w;
          }
      }
    }
#pragma unroll
    for (int j = 0; j < J; ++j) {
      const int it = it0 + j * nt;
      if (it >= items) continue;
      const int qi = it / c4n, c = (it % c4n) * 4;
      const size_t o = static_cast<size_t>(b * p.q_rows + qi) * p.ldo + h * hd + c;
      store_act4(out, out_lo, o, acc[j]);
    }
  }
}

template <typename TKV, typename T, int HD>
__global__ void __launch_bounds__(WARPS * 32) attn_kernel(const AttnParams p) {
  pdl_trigger();  // the next kernel may start its prologue
  pdl_wait();     // inputs of this kernel are complete
  // SIMT path: fp32 models and bf16 models with head_dim 64
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
        const TKV* base = pool + (static_cast<size_t>(page) * p.H + h) * p.planes * 16 * HD + (key & 15) * HD + dd;
        const int vp = p.planes / 2;
        kv = to_f(base[0]);
        vv = to_f(base[vp * 16 * HD]);
        if (p.planes == 4) {
          kv += to_f(base[16 * HD]);
          vv += to_f(base[3 * 16 * HD]);
        }
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

  const size_t rec = HD + 4;
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
  combine_splits(p, wsb, nq, HD, b, h, out, out_lo, sm);  // the K/V tile area is free now
  if (threadIdx.x == 0) p.counters[b * p.H + h] = 0;
}

constexpr int ATT_MAX_DEVICES = 64;
std::mutex g_attr_mu;

template <typename TKV, typename T, int HD>
cudaError_t launch(const AttnParams& p, cudaStream_t s) {
  const size_t smem = (KT * (HD + 1) + KT * HD + static_cast<size_t>(p.nq_max) * HD) * sizeof(float);
  // the shared-memory limit is a per-device attribute: raised once per device
  static bool attr[ATT_MAX_DEVICES];
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= ATT_MAX_DEVICES) return cudaErrorInvalidDevice;
  {
    std::lock_guard<std::mutex> lk(g_attr_mu);
    if (!attr[dev]) {
      e = cudaFuncSetAttribute(attn_kernel<TKV, T, HD>, cudaFuncAttributeMaxDynamicSharedMemorySize, 200 * 1024);
      if (e != cudaSuccess) return e;
      attr[dev] = true;
    }
  }
  dim3 grid(p.splits, p.H, p.B);
  launch_pdl(attn_kernel<TKV, T, HD>, dim3(grid), dim3(WARPS * 32), smem, s, p);
  return cudaGetLastError();
}

}  // namespace

size_t attn_ws_floats(int B, int H, int splits, int nq_max, int hd) {
  return static_cast<size_t>(B) * H * splits * nq_max * (hd + 4);
}

bool attn_fuses_rope(int dtype, int hd) { return dtype == 1 && hd == 128; }

int attn_pick_splits(int dtype, int hd, int planes, int B, int H, int want) {
  if (!attn_fuses_rope(dtype, hd)) return want;
  return attention_tc_splits(planes, B * H, want);
}

cudaError_t attention(const AttnParams& p, int dtype, cudaStream_t s) {
  if (p.nq_max > WARPS * QPW || p.n_local > 64 || p.splits > MAX_SPLITS || p.splits < 1) return cudaErrorInvalidValue;
  if (p.planes != 2 && !(p.planes == 4 && dtype == 1)) return cudaErrorInvalidValue;
  if (dtype == 0) {
    if (p.qkv) return cudaErrorInvalidValue;
    if (p.hd == 64) return launch<float, float, 64>(p, s);
    if (p.hd == 128) return launch<float, float, 128>(p, s);
  } else if (p.hd == 128) {
    if (p.splits > 8) return cudaErrorInvalidValue;  // one cluster of at most 8 CTAs per (b, h)
    if (p.qkv && (!p.rope || !p.err || p.max_pos < 1 || (p.ldqkv & 3))) return cudaErrorInvalidValue;
    return attention_tc(p, s);
  } else if (p.hd == 64) {
    if (p.qkv) return cudaErrorInvalidValue;
    return launch<bf16, bf16, 64>(p, s);
  }
  return cudaErrorInvalidValue;
}

}  // namespace chimera
