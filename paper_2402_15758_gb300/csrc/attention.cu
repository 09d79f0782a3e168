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
// into shared memory for all the sequence's queries; online softmax in fp32.  With
// several splits, every CTA writes (unnormalised output, running max, running sum)
// and the last CTA of the (b, h) pair merges them in split order.
#include <cmath>

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
      store_act(out, out_lo, o, acc[j].x);
      store_act(out, out_lo, o + 1, acc[j].y);
      store_act(out, out_lo, o + 2, acc[j].z);
      store_act(out, out_lo, o + 3, acc[j].w);
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

// ---------------------------------------------------------------------------
// Tensor-core path for bf16 models (head_dim 128): QK^T and PV on mma.sync
// m16n8k16 with fp32 accumulation.  Every bf16 operand is a two-term split of the
// fp32 value (x = hi + lo); each product takes the three terms hi*hi + hi*lo + lo*hi,
// so the result matches fp32 arithmetic to ~2^-16.  KV tiles of 64 keys are staged
// in shared memory as bf16 hi/lo planes (padded rows, ldmatrix-friendly); each warp
// owns 16 queries.
// ---------------------------------------------------------------------------
#ifdef CHIMERA_ATTN_TRACE
// per-CTA timestamps of the last launch (instrumented builds only)
__device__ unsigned long long g_attn_trace[2048][8];
#define ATRACE(i) \
  if (threadIdx.x == 0) g_attn_trace[(blockIdx.z * gridDim.y + blockIdx.y) * gridDim.x + blockIdx.x][i] = global_timer_ns()
#else
#define ATRACE(i)
#endif

constexpr int MKT = 64;              // keys per tile
constexpr int MHD = 128;             // head dim
constexpr int MLDS = MHD + 8;        // smem row pitch (bf16): 272 B, conflict-free ldmatrix
constexpr int MWARPS = 8;

__device__ __forceinline__ uint32_t pack_bf16(bf16 a, bf16 b) {
  return static_cast<uint32_t>(__bfloat16_as_ushort(a)) | (static_cast<uint32_t>(__bfloat16_as_ushort(b)) << 16);
}
// (x, y) -> hi pair and lo pair
__device__ __forceinline__ void split2(float x, float y, uint32_t& hi, uint32_t& lo) {
  const bf16 hx = __float2bfloat16_rn(x), hy = __float2bfloat16_rn(y);
  hi = pack_bf16(hx, hy);
  lo = pack_bf16(__float2bfloat16_rn(x - __bfloat162float(hx)), __float2bfloat16_rn(y - __bfloat162float(hy)));
}
// Not volatile: a pure register operation, so the compiler may interleave independent
// accumulator chains.
__device__ __forceinline__ void mma16816(float (&d)[4], const uint32_t (&a)[4], uint32_t b0, uint32_t b1) {
  asm(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
      "{%0,%1,%2,%3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}
__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2, uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}
__device__ __forceinline__ void ldsm_x4_t(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2, uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}

__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src, bool valid) {
  // 16-byte async copy; src_size 0 fills the destination with zeros
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst), "l"(src), "r"(valid ? 16 : 0)
               : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
__device__ __forceinline__ void cp_async_wait1() { asm volatile("cp.async.wait_group 1;" ::: "memory"); }

// SPLIT: the cache holds K_hi, K_lo, V_hi, V_lo planes (three-term products);
// otherwise K, V planes (K_lo = V_lo = 0: two-term products for the split queries and P).
// 8 warps: warp w owns queries 16*(w & 3) .. +15 and the key half (w >> 2) of every
// 64-key tile; the two halves' online-softmax states merge at the end.
template <bool SPLIT>
__global__ void __launch_bounds__(MWARPS * 32) attn_mma_kernel(const AttnParams p) {
  pdl_trigger();  // the next kernel may start its prologue
  pdl_wait();     // inputs of this kernel are complete
  constexpr int NP = SPLIT ? 4 : 2;                  // planes per (block, head)
  constexpr int STAGE = NP * MKT * MLDS;             // bf16 elements per pipeline stage
  extern __shared__ __align__(16) uint8_t smem_raw[];
  bf16* stage_base = reinterpret_cast<bf16*>(smem_raw);
  __shared__ int s_last;

  const int s = blockIdx.x, h = blockIdx.y, b = blockIdx.z;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int qg = warp & 3, kh = warp >> 2;
  ATRACE(0);
  const int nctx = p.n_ctx[b];
  const int nloc = p.n_local_dev ? p.n_local_dev[b] : p.n_local;
  const int nq = p.nq_dev ? p.nq_dev[b] : p.nq;
  const int total = nctx + nloc;
  const int ntiles = (total + MKT - 1) / MKT;
  const int tps = (ntiles + p.splits - 1) / p.splits;
  const int t0 = s * tps;
  const int t1 = min(ntiles, t0 + tps);
  const bf16* pool = static_cast<const bf16*>(p.pool) + static_cast<size_t>(p.layer) * p.pool_layer_stride;

  // staging: thread copies 16-byte chunk (tid & 15) of key row (tid >> 4) + 16u of every
  // plane, u = 0..3 (one 16-key page each); keys past the end are zero-filled
  const int krow = threadIdx.x >> 4, kch = threadIdx.x & 15;
  auto issue_tile = [&](int t, int st) {
    const uint32_t sbase = smem_u32(stage_base + st * STAGE);
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const int kg = t * MKT + u * 16 + krow;
      const bool valid = kg < total;
      const bf16* src = pool;
      if (valid) {
        const int page = p.page_table[b * p.max_pages + t * 4 + u];
        src = pool + (static_cast<size_t>(page) * p.H + h) * NP * 16 * MHD + krow * MHD + kch * 8;
      }
#pragma unroll
      for (int plane = 0; plane < NP; ++plane)
        cp_async16(sbase + static_cast<uint32_t>(((plane * MKT + u * 16 + krow) * MLDS + kch * 8) * 2),
                   valid ? src + plane * 16 * MHD : src, valid);
    }
    cp_async_commit();
  };

  const int qw = qg * 16;
  const bool active = qw < nq;
  const int r0 = qw + (lane >> 2), r1 = r0 + 8;
  const int cq = (lane & 3) * 2;

  // query fragments (A operand, row-major 16 x 128), hi and lo halves
  uint32_t qh[8][4], ql[8][4];
#pragma unroll
  for (int ks = 0; ks < 8; ++ks) {
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int row = (j & 1) ? r1 : r0;
      const int col = ks * 16 + cq + ((j & 2) ? 8 : 0);
      float x = 0.f, y = 0.f;
      if (row < nq) {
        const float2 v = *reinterpret_cast<const float2*>(p.q + static_cast<size_t>(b * p.q_rows + row) * p.ldq + h * MHD + col);
        x = v.x; y = v.y;
      }
      split2(x, y, qh[ks][j], ql[ks][j]);
    }
  }
  const unsigned long long m0 = r0 < nq ? p.anc[p.q_local0 + r0] : 0ull;
  const unsigned long long m1 = r1 < nq ? p.anc[p.q_local0 + r1] : 0ull;

  float o[16][4];
#pragma unroll
  for (int i = 0; i < 16; ++i) o[i][0] = o[i][1] = o[i][2] = o[i][3] = 0.f;
  float mrow[2] = {-INFINITY, -INFINITY}, lrow[2] = {0.f, 0.f};
  ATRACE(1);

  if (t0 < t1) issue_tile(t0, 0);
  for (int t = t0; t < t1; ++t) {
    const int st = (t - t0) & 1;
    if (t + 1 < t1)
      issue_tile(t + 1, st ^ 1);  // the other stage was released by the barrier below
    else
      cp_async_commit();
    cp_async_wait1();
    __syncthreads();
    if (t == t0) ATRACE(2);
    if (active) {
      const uint32_t kh_base = smem_u32(stage_base + st * STAGE);
      const uint32_t kl_base = kh_base + (SPLIT ? MKT * MLDS * 2 : 0);
      const uint32_t vh_base = kh_base + (SPLIT ? 2 : 1) * MKT * MLDS * 2;
      const uint32_t vl_base = vh_base + (SPLIT ? MKT * MLDS * 2 : 0);
      // S = Q K^T on this warp's 32 keys (4 n-tiles of 8)
      float sc[4][4];
#pragma unroll
      for (int nt = 0; nt < 4; ++nt) sc[nt][0] = sc[nt][1] = sc[nt][2] = sc[nt][3] = 0.f;
#pragma unroll
      for (int kp = 0; kp < 4; ++kp) {  // 32 dims per ldmatrix.x4 = two k-steps
#pragma unroll
        for (int nt = 0; nt < 4; ++nt) {
          const uint32_t roff =
              static_cast<uint32_t>((((kh * 4 + nt) * 8 + (lane & 7)) * MLDS + (lane >> 3) * 8) * 2);
          uint32_t bh0, bh1, bh2, bh3;
          ldsm_x4(kh_base + roff + kp * 64, bh0, bh1, bh2, bh3);
          mma16816(sc[nt], qh[2 * kp], bh0, bh1);
          mma16816(sc[nt], ql[2 * kp], bh0, bh1);
          mma16816(sc[nt], qh[2 * kp + 1], bh2, bh3);
          mma16816(sc[nt], ql[2 * kp + 1], bh2, bh3);
          if (SPLIT) {
            uint32_t bl0, bl1, bl2, bl3;
            ldsm_x4(kl_base + roff + kp * 64, bl0, bl1, bl2, bl3);
            mma16816(sc[nt], qh[2 * kp], bl0, bl1);
            mma16816(sc[nt], qh[2 * kp + 1], bl2, bl3);
          }
        }
      }
      // mask, scale, online softmax (rows r0: elements 0,1; r1: elements 2,3)
      float tmax[2] = {-INFINITY, -INFINITY};
#pragma unroll
      for (int nt = 0; nt < 4; ++nt) {
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const int key = t * MKT + (kh * 4 + nt) * 8 + cq + (e & 1);
          const unsigned long long m = (e < 2) ? m0 : m1;
          const bool vis = key < nctx || (key < total && ((m >> (key - nctx)) & 1ull));
          sc[nt][e] = vis ? sc[nt][e] * p.scale : -INFINITY;
          tmax[e >> 1] = fmaxf(tmax[e >> 1], sc[nt][e]);
        }
      }
      float corr[2];
#pragma unroll
      for (int r = 0; r < 2; ++r) {
        tmax[r] = fmaxf(tmax[r], __shfl_xor_sync(0xffffffffu, tmax[r], 1));
        tmax[r] = fmaxf(tmax[r], __shfl_xor_sync(0xffffffffu, tmax[r], 2));
        const float mnew = fmaxf(mrow[r], tmax[r]);
        corr[r] = (mnew == -INFINITY) ? 1.f : expf(mrow[r] - mnew);
        mrow[r] = mnew;
      }
      float rsum[2] = {0.f, 0.f};
#pragma unroll
      for (int nt = 0; nt < 4; ++nt) {
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const float pv = (sc[nt][e] == -INFINITY) ? 0.f : expf(sc[nt][e] - mrow[e >> 1]);
          sc[nt][e] = pv;
          rsum[e >> 1] += pv;
        }
      }
#pragma unroll
      for (int r = 0; r < 2; ++r) {
        rsum[r] += __shfl_xor_sync(0xffffffffu, rsum[r], 1);
        rsum[r] += __shfl_xor_sync(0xffffffffu, rsum[r], 2);
        lrow[r] = lrow[r] * corr[r] + rsum[r];
      }
#pragma unroll
      for (int dt = 0; dt < 16; ++dt) {
        o[dt][0] *= corr[0]; o[dt][1] *= corr[0];
        o[dt][2] *= corr[1]; o[dt][3] *= corr[1];
      }
      // O += P V over this warp's 32 keys: two k-steps of 16 keys, 16 n-tiles of 8 dims
#pragma unroll
      for (int kk = 0; kk < 2; ++kk) {
        uint32_t ph[4], pl[4];
        split2(sc[2 * kk][0], sc[2 * kk][1], ph[0], pl[0]);
        split2(sc[2 * kk][2], sc[2 * kk][3], ph[1], pl[1]);
        split2(sc[2 * kk + 1][0], sc[2 * kk + 1][1], ph[2], pl[2]);
        split2(sc[2 * kk + 1][2], sc[2 * kk + 1][3], ph[3], pl[3]);
        // ldmatrix.trans rows: key kh*32 + kk*16 + (lane & 15), dims 8 * (lane >> 4)
        const uint32_t roff =
            static_cast<uint32_t>(((kh * 32 + kk * 16 + (lane & 15)) * MLDS + (lane >> 4) * 8) * 2);
#pragma unroll
        for (int dp = 0; dp < 8; ++dp) {  // two n-tiles per ldmatrix.x4
          uint32_t vh0, vh1, vh2, vh3;
          ldsm_x4_t(vh_base + roff + dp * 32, vh0, vh1, vh2, vh3);
          mma16816(o[2 * dp], ph, vh0, vh1);
          mma16816(o[2 * dp], pl, vh0, vh1);
          mma16816(o[2 * dp + 1], ph, vh2, vh3);
          mma16816(o[2 * dp + 1], pl, vh2, vh3);
          if (SPLIT) {
            uint32_t vl0, vl1, vl2, vl3;
            ldsm_x4_t(vl_base + roff + dp * 32, vl0, vl1, vl2, vl3);
            mma16816(o[2 * dp], ph, vl0, vl1);
            mma16816(o[2 * dp + 1], ph, vl2, vl3);
          }
        }
      }
    }
    __syncthreads();  // this stage may be refilled by the next iteration's copies
  }

  ATRACE(3);
  // merge the two key halves: warps 4..7 hand their state to warps 0..3 (same lane,
  // same query rows and dims)
  float* xch = reinterpret_cast<float*>(smem_raw);  // [4 groups][32 lanes][68]
  if (kh == 1 && active) {
    float* x = xch + (qg * 32 + lane) * 68;
#pragma unroll
    for (int dt = 0; dt < 16; ++dt)
#pragma unroll
      for (int e = 0; e < 4; ++e) x[dt * 4 + e] = o[dt][e];
    x[64] = mrow[0]; x[65] = mrow[1]; x[66] = lrow[0]; x[67] = lrow[1];
  }
  __syncthreads();
  if (kh == 0 && active) {
    const float* x = xch + (qg * 32 + lane) * 68;
#pragma unroll
    for (int r = 0; r < 2; ++r) {
      const float mb = x[64 + r], lb = x[66 + r];
      const float M = fmaxf(mrow[r], mb);
      const float ca = (M == -INFINITY) ? 0.f : expf(mrow[r] - M);
      const float cb = (M == -INFINITY) ? 0.f : expf(mb - M);
      lrow[r] = lrow[r] * ca + lb * cb;
      mrow[r] = M;
#pragma unroll
      for (int dt = 0; dt < 16; ++dt) {
        o[dt][2 * r] = o[dt][2 * r] * ca + x[dt * 4 + 2 * r] * cb;
        o[dt][2 * r + 1] = o[dt][2 * r + 1] * ca + x[dt * 4 + 2 * r + 1] * cb;
      }
    }
  }
  const bool writer = kh == 0 && active;

  bf16* out = static_cast<bf16*>(p.out);
  bf16* out_lo = static_cast<bf16*>(p.out_lo);
  if (p.splits == 1) {
    if (!writer) return;
#pragma unroll
    for (int r = 0; r < 2; ++r) {
      const int row = r ? r1 : r0;
      if (row >= nq) continue;
      const float inv = lrow[r] > 0.f ? 1.f / lrow[r] : 0.f;
      const size_t base = static_cast<size_t>(b * p.q_rows + row) * p.ldo + h * MHD + cq;
#pragma unroll
      for (int dt = 0; dt < 16; ++dt) {
        store_act(out, out_lo, base + dt * 8, o[dt][2 * r] * inv);
        store_act(out, out_lo, base + dt * 8 + 1, o[dt][2 * r + 1] * inv);
      }
    }
    return;
  }

  const size_t rec = MHD + 4;
  float* wsb = p.ws + (static_cast<size_t>(b * p.H + h) * p.splits) * p.nq_max * rec;
  if (writer) {
#pragma unroll
    for (int r = 0; r < 2; ++r) {
      const int row = r ? r1 : r0;
      if (row >= nq) continue;
      float* w = wsb + (static_cast<size_t>(s) * p.nq_max + row) * rec;
#pragma unroll
      for (int dt = 0; dt < 16; ++dt) {
        __stcg(&w[dt * 8 + cq], o[dt][2 * r]);
        __stcg(&w[dt * 8 + cq + 1], o[dt][2 * r + 1]);
      }
      if ((lane & 3) == 0) {
        __stcg(&w[MHD], mrow[r]);
        __stcg(&w[MHD + 1], lrow[r]);
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
  ATRACE(4);
  if (!s_last) return;
  __threadfence();
  combine_splits(p, wsb, nq, MHD, b, h, out, out_lo, reinterpret_cast<float*>(smem_raw));
  if (threadIdx.x == 0) p.counters[b * p.H + h] = 0;
  ATRACE(5);
}

template <bool SPLIT>
cudaError_t launch_mma(const AttnParams& p, cudaStream_t s) {
  const size_t smem = 2 * (SPLIT ? 4 : 2) * MKT * MLDS * sizeof(bf16);  // two pipeline stages
  static bool attr = false;
  if (!attr) {
    cudaFuncSetAttribute(attn_mma_kernel<SPLIT>, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
    attr = true;
  }
  dim3 grid(p.splits, p.H, p.B);
  launch_pdl(attn_mma_kernel<SPLIT>, dim3(grid), dim3(MWARPS * 32), smem, s, p);
  return cudaGetLastError();
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
  launch_pdl(attn_kernel<TKV, T, HD>, dim3(grid), dim3(WARPS * 32), smem, s, p);
  return cudaGetLastError();
}

}  // namespace

#ifdef CHIMERA_ATTN_TRACE
extern "C" int chimera_attn_trace(unsigned long long* host, int n) {
  return cudaMemcpyFromSymbol(host, g_attn_trace, static_cast<size_t>(n) * 8 * 8) == cudaSuccess ? 0 : -1;
}
#endif

size_t attn_ws_floats(int B, int H, int splits, int nq_max, int hd) {
  return static_cast<size_t>(B) * H * splits * nq_max * (hd + 4);
}

cudaError_t attention(const AttnParams& p, int dtype, cudaStream_t s) {
  if (p.nq_max > WARPS * QPW || p.n_local > 64 || p.splits > MAX_SPLITS) return cudaErrorInvalidValue;
  if (p.planes != 2 && !(p.planes == 4 && dtype == 1)) return cudaErrorInvalidValue;
  if (dtype == 0) {
    if (p.hd == 64) return launch<float, float, 64>(p, s);
    if (p.hd == 128) return launch<float, float, 128>(p, s);
  } else if (p.hd == 128) {
    return p.planes == 4 ? launch_mma<true>(p, s) : launch_mma<false>(p, s);
  } else if (p.hd == 64) {
    return launch<bf16, bf16, 64>(p, s);
  }
  return cudaErrorInvalidValue;
}

}  // namespace chimera
