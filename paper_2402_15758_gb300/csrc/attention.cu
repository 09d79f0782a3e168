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
// into shared memory for all the sequence's queries; online softmax in fp32.  Two
// kernels: a SIMT one (fp32 models, head_dim 64) whose splits merge in the last CTA of
// each (b, h) through a global workspace, and a tensor-core one (bf16, head_dim 128)
// whose splits form a thread-block cluster and merge through distributed shared
// memory; the latter can also apply RoPE to q and to the step's fresh k rows and write
// their k, v into the cache (the fused mode used by the step).
#include <algorithm>
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

__device__ __forceinline__ void cp_async_wait0() { asm volatile("cp.async.wait_group 0;" ::: "memory"); }
__device__ __forceinline__ void cp_async_wait2() { asm volatile("cp.async.wait_group 2;" ::: "memory"); }

constexpr int TREE_STAGES = 3;         // KV tiles in the ring
constexpr int TREE_PAGE_CACHE = 1024;  // page indices cached per CTA (256 tiles)

// SPLIT: the cache holds K_hi, K_lo, V_hi, V_lo planes (three-term products);
// otherwise K, V planes (K_lo = V_lo = 0: two-term products for the split queries and P).
//
// Grid (S, H, B), one thread-block cluster of S CTAs per (b, h).  CTA s takes the
// contiguous 64-key tiles [t0, t1) of the sequence's keys; 8 warps: warp w owns queries
// 16*(w & 3) .. +15 and the key half (w >> 2) of every tile, the two halves merge in
// shared memory, and the S partial states (unnormalised output, running max, running
// sum) merge across the cluster through distributed shared memory: CTA r finishes the
// query rows [r * ceil(nq / S), ...).  KV tiles stream through a three-stage cp.async
// ring (two tiles in flight while one is consumed); the CTA's page indices are cached
// in shared memory, and committed-context tiles may be requested before the kernel's
// dependency wait.
template <bool SPLIT>
__global__ void __launch_bounds__(MWARPS * 32, 1) attn_tree_kernel(const AttnParams p) {
  constexpr int NP = SPLIT ? 4 : 2;                  // planes per (block, head)
  constexpr int STAGE = NP * MKT * MLDS;             // bf16 elements per pipeline stage
  constexpr int PREC = MHD + 4;                      // partial record: o[128], m, l, pad
  extern __shared__ __align__(16) uint8_t smem_raw[];
  __shared__ int s_pages[TREE_PAGE_CACHE];
  bf16* stage_base = reinterpret_cast<bf16*>(smem_raw);
  float* xch = reinterpret_cast<float*>(smem_raw);                  // [4][32][68] key-half merge
  float* part = reinterpret_cast<float*>(smem_raw) + 4 * 32 * 68;   // [64][PREC] cluster merge

  const int s = blockIdx.x, h = blockIdx.y, b = blockIdx.z;
  const int S = gridDim.x;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int qg = warp & 3, kh = warp >> 2;
  ATRACE(0);
  bf16* pool = static_cast<bf16*>(const_cast<void*>(p.pool)) + static_cast<size_t>(p.layer) * p.pool_layer_stride;

  if (!p.prewait_kv) pdl_wait();
  const int nctx = p.n_ctx[b];
  // the tile partition uses the launch's maximum local count, so it is known before
  // the wait; keys past the sequence's real end are masked
  const int ntiles = (nctx + p.n_local + MKT - 1) / MKT;
  const int tps = (ntiles + S - 1) / S;
  const int t0 = min(ntiles, s * tps);
  const int t1 = min(ntiles, t0 + tps);
  // page indices of the CTA's pages (the table is not written during a step)
  const bool cached = (t1 - t0) * 4 <= TREE_PAGE_CACHE;
  if (cached) {
    const int np = min((t1 - t0) * 4, p.max_pages - t0 * 4);
    for (int i = threadIdx.x; i < np; i += blockDim.x) s_pages[i] = p.page_table[b * p.max_pages + t0 * 4 + i];
  }
  __syncthreads();

  // staging: thread copies 16-byte chunk (tid & 15) of key row (tid >> 4) + 16u of every
  // plane, u = 0..3 (one 16-key page each); keys at or past kend are zero-filled
  const int krow = threadIdx.x >> 4, kch = threadIdx.x & 15;
  auto issue_tile = [&](int t, int st, int kend) {
    const uint32_t sbase = smem_u32(stage_base + st * STAGE);
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const int kg = t * MKT + u * 16 + krow;
      const bool valid = kg < kend;
      const bf16* src = pool;
      if (valid) {
        const int page = cached ? s_pages[(t - t0) * 4 + u] : p.page_table[b * p.max_pages + t * 4 + u];
        src = pool + (static_cast<size_t>(page) * p.H + h) * NP * 16 * MHD + krow * MHD + kch * 8;
      }
#pragma unroll
      for (int plane = 0; plane < NP; ++plane)
        cp_async16(sbase + static_cast<uint32_t>(((plane * MKT + u * 16 + krow) * MLDS + kch * 8) * 2),
                   valid ? src + plane * 16 * MHD : src, valid);
    }
    cp_async_commit();
  };

  // committed-context tiles do not depend on the preceding kernels of this step
  int issued = t0;
  if (p.prewait_kv) {
    while (issued < t1 && issued < t0 + TREE_STAGES && (issued + 1) * MKT <= nctx) {
      issue_tile(issued, issued - t0, nctx);
      ++issued;
    }
    pdl_wait();
  }
  pdl_trigger();  // after the wait: a dependent may rely on every earlier kernel being complete

  const int nloc = min(p.n_local_dev ? p.n_local_dev[b] : p.n_local, p.n_local);
  const int nq = p.nq_dev ? p.nq_dev[b] : p.nq;
  const int total = nctx + nloc;

  const int qw = qg * 16;
  const bool active = qw < nq;
  const int r0 = qw + (lane >> 2), r1 = r0 + 8;
  const int cq = (lane & 3) * 2;
  const int dm = p.H * MHD;

  if (p.qkv) {
    // fresh local rows inside this CTA's key range: rotate k, write k and v (hi/lo
    // planes) into the pool; the tiles below read them back
    const int fresh0 = nctx + p.q_local0;
    const int f0 = max(0, t0 * MKT - fresh0), f1 = min(nq, t1 * MKT - fresh0);
    for (int it = threadIdx.x; it < (f1 - f0) * 16; it += blockDim.x) {
      const int i = f0 + (it >> 4), j = (it & 15) * 4;
      const int slot = fresh0 + i;
      const int pos = nctx + p.pos_base + (p.pos_off ? p.pos_off[i] : i);
      if (pos < 0 || pos >= p.max_pos || (slot >> 4) >= p.max_pages) {
        atomicOr(p.err, ERR_CAPACITY);
        continue;
      }
      const int page = p.page_table[b * p.max_pages + (slot >> 4)];
      const float* src = p.qkv + static_cast<size_t>(b * p.q_rows + i) * p.ldqkv + h * MHD + j;
      const float4 k1 = *reinterpret_cast<const float4*>(src + dm);
      const float4 k2 = *reinterpret_cast<const float4*>(src + dm + MHD / 2);
      const float4 v1 = *reinterpret_cast<const float4*>(src + 2 * dm);
      const float4 v2 = *reinterpret_cast<const float4*>(src + 2 * dm + MHD / 2);
      const float2* tab = p.rope + static_cast<size_t>(pos) * (MHD / 2) + j;
      const float4 cs01 = *reinterpret_cast<const float4*>(tab);
      const float4 cs23 = *reinterpret_cast<const float4*>(tab + 2);
      const float4 c = make_float4(cs01.x, cs01.z, cs23.x, cs23.z);
      const float4 sn = make_float4(cs01.y, cs01.w, cs23.y, cs23.w);
      const float4 ka = rot_lo(k1, k2, c, sn), kb = rot_hi(k1, k2, c, sn);
      bf16* base = pool + (static_cast<size_t>(page) * p.H + h) * NP * 16 * MHD + (slot & 15) * MHD + j;
      constexpr size_t plane = 16 * MHD;
      if (SPLIT) {
        store4_split(base, base + plane, ka);
        store4_split(base + MHD / 2, base + plane + MHD / 2, kb);
        store4_split(base + 2 * plane, base + 3 * plane, v1);
        store4_split(base + 2 * plane + MHD / 2, base + 3 * plane + MHD / 2, v2);
      } else {
        store4<bf16>(base, ka);
        store4<bf16>(base + MHD / 2, kb);
        store4<bf16>(base + plane, v1);
        store4<bf16>(base + plane + MHD / 2, v2);
      }
    }
    __threadfence_block();
    __syncthreads();
  }
  while (issued < t1 && issued < t0 + TREE_STAGES) {
    issue_tile(issued, issued - t0, total);
    ++issued;
  }

  // query fragments (A operand, row-major 16 x 128), hi and lo halves; in the fused
  // mode q is rotated here (pairs (c, c + 64) sit in fragments ks and ks + 4)
  uint32_t qh[8][4], ql[8][4];
  if (p.qkv) {
    const float2* tab0 = nullptr;
    const float2* tab1 = nullptr;
    if (r0 < nq) {
      const int pos = min(max(nctx + p.pos_base + (p.pos_off ? p.pos_off[r0] : r0), 0), p.max_pos - 1);
      tab0 = p.rope + static_cast<size_t>(pos) * (MHD / 2);
    }
    if (r1 < nq) {
      const int pos = min(max(nctx + p.pos_base + (p.pos_off ? p.pos_off[r1] : r1), 0), p.max_pos - 1);
      tab1 = p.rope + static_cast<size_t>(pos) * (MHD / 2);
    }
#pragma unroll
    for (int ks = 0; ks < 4; ++ks) {
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const int row = (j & 1) ? r1 : r0;
        const float2* tab = (j & 1) ? tab1 : tab0;
        const int col = ks * 16 + cq + ((j & 2) ? 8 : 0);
        float x0 = 0.f, x1 = 0.f, y0 = 0.f, y1 = 0.f;
        if (row < nq) {
          const float* src = p.qkv + static_cast<size_t>(b * p.q_rows + row) * p.ldqkv + h * MHD + col;
          const float2 a = *reinterpret_cast<const float2*>(src);
          const float2 a2 = *reinterpret_cast<const float2*>(src + MHD / 2);
          const float4 cs = *reinterpret_cast<const float4*>(tab + col);  // (cos, sin) of col, col + 1
          x0 = a.x * cs.x - a2.x * cs.y;
          x1 = a.y * cs.z - a2.y * cs.w;
          y0 = a2.x * cs.x + a.x * cs.y;
          y1 = a2.y * cs.z + a.y * cs.w;
        }
        split2(x0, x1, qh[ks][j], ql[ks][j]);
        split2(y0, y1, qh[ks + 4][j], ql[ks + 4][j]);
      }
    }
  } else {
#pragma unroll
    for (int ks = 0; ks < 8; ++ks) {
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const int row = (j & 1) ? r1 : r0;
        const int col = ks * 16 + cq + ((j & 2) ? 8 : 0);
        float x = 0.f, y = 0.f;
        if (row < nq) {
          const float2 v =
              *reinterpret_cast<const float2*>(p.q + static_cast<size_t>(b * p.q_rows + row) * p.ldq + h * MHD + col);
          x = v.x;
          y = v.y;
        }
        split2(x, y, qh[ks][j], ql[ks][j]);
      }
    }
  }
  const unsigned long long m0 = r0 < nq ? p.anc[p.q_local0 + r0] : 0ull;
  const unsigned long long m1 = r1 < nq ? p.anc[p.q_local0 + r1] : 0ull;

  float o[16][4];
#pragma unroll
  for (int i = 0; i < 16; ++i) o[i][0] = o[i][1] = o[i][2] = o[i][3] = 0.f;
  float mrow[2] = {-INFINITY, -INFINITY}, lrow[2] = {0.f, 0.f};
  ATRACE(1);

  for (int t = t0; t < t1; ++t) {
    const int st = (t - t0) % TREE_STAGES;
    // tiles t .. issued-1 are in flight: let the newer ones stay pending
    if (issued - t >= 3)
      cp_async_wait2();
    else if (issued - t == 2)
      cp_async_wait1();
    else
      cp_async_wait0();
    __syncthreads();
    if (t == t0) ATRACE(2);
    if (active) {
      const uint32_t kh_base = smem_u32(stage_base + st * STAGE);
      const uint32_t kl_base = kh_base + (SPLIT ? MKT * MLDS * 2 : 0);
      const uint32_t vh_base = kh_base + (SPLIT ? 2 : 1) * MKT * MLDS * 2;
      const uint32_t vl_base = vh_base + (SPLIT ? MKT * MLDS * 2 : 0);
      // S = Q K^T on this warp's 32 keys (4 n-tiles of 8); the three product terms
      // accumulate separately (independent MMA chains), summed after the loop
      float sa[4][4], sb[4][4], sc2[4][4];
#pragma unroll
      for (int nt = 0; nt < 4; ++nt)
#pragma unroll
        for (int e = 0; e < 4; ++e) sa[nt][e] = sb[nt][e] = sc2[nt][e] = 0.f;
#pragma unroll
      for (int kp = 0; kp < 4; ++kp) {  // 32 dims per ldmatrix.x4 = two k-steps
#pragma unroll
        for (int nt = 0; nt < 4; ++nt) {
          const uint32_t roff =
              static_cast<uint32_t>((((kh * 4 + nt) * 8 + (lane & 7)) * MLDS + (lane >> 3) * 8) * 2);
          uint32_t bh0, bh1, bh2, bh3;
          ldsm_x4(kh_base + roff + kp * 64, bh0, bh1, bh2, bh3);
          mma16816(sa[nt], qh[2 * kp], bh0, bh1);
          mma16816(sb[nt], ql[2 * kp], bh0, bh1);
          mma16816(sa[nt], qh[2 * kp + 1], bh2, bh3);
          mma16816(sb[nt], ql[2 * kp + 1], bh2, bh3);
          if (SPLIT) {
            uint32_t bl0, bl1, bl2, bl3;
            ldsm_x4(kl_base + roff + kp * 64, bl0, bl1, bl2, bl3);
            mma16816(sc2[nt], qh[2 * kp], bl0, bl1);
            mma16816(sc2[nt], qh[2 * kp + 1], bl2, bl3);
          }
        }
      }
      float sc[4][4];
      // mask, scale, online softmax (rows r0: elements 0,1; r1: elements 2,3)
      float tmax[2] = {-INFINITY, -INFINITY};
#pragma unroll
      for (int nt = 0; nt < 4; ++nt) {
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const int key = t * MKT + (kh * 4 + nt) * 8 + cq + (e & 1);
          const unsigned long long m = (e < 2) ? m0 : m1;
          const bool vis = key < nctx || (key < total && ((m >> (key - nctx)) & 1ull));
          const float dot = (sa[nt][e] + sb[nt][e]) + sc2[nt][e];
          sc[nt][e] = vis ? dot * p.scale : -INFINITY;
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
          mma16816(o[2 * dp + 1], ph, vh2, vh3);
          mma16816(o[2 * dp], pl, vh0, vh1);
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
    __syncthreads();  // this stage may be refilled now
    if (issued < t1) {
      issue_tile(issued, (issued - t0) % TREE_STAGES, total);
      ++issued;
    }
  }

  ATRACE(3);
  // merge the two key halves: warps 4..7 hand their state to warps 0..3 (same lane,
  // same query rows and dims)
  if (kh == 1 && active) {
    float* x = xch + (qg * 32 + lane) * 68;
#pragma unroll
    for (int dt = 0; dt < 16; ++dt)
#pragma unroll
      for (int e = 0; e < 4; ++e) x[dt * 4 + e] = o[dt][e];
    x[64] = mrow[0]; x[65] = mrow[1]; x[66] = lrow[0]; x[67] = lrow[1];
  }
  __syncthreads();
  const bool writer = kh == 0 && active;
  if (writer) {
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

  bf16* out = static_cast<bf16*>(p.out);
  bf16* out_lo = static_cast<bf16*>(p.out_lo);
  if (S == 1) {
    if (writer) {
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
    }
    return;
  }

  // cluster merge: every CTA publishes its partial rows, CTA s finishes its share
  if (writer) {
#pragma unroll
    for (int r = 0; r < 2; ++r) {
      const int row = r ? r1 : r0;
      if (row >= nq) continue;
      float* w = part + row * PREC;
#pragma unroll
      for (int dt = 0; dt < 16; ++dt) {
        w[dt * 8 + cq] = o[dt][2 * r];
        w[dt * 8 + cq + 1] = o[dt][2 * r + 1];
      }
      if ((lane & 3) == 0) {
        w[MHD] = mrow[r];
        w[MHD + 1] = lrow[r];
      }
    }
  }
  cluster_sync();
  ATRACE(4);
  {
    const int rpc = (nq + S - 1) / S;
    const int q0 = s * rpc, q1 = min(nq, q0 + rpc);
    const uint32_t part_u32 = smem_u32(part);
    for (int it = threadIdx.x; it < (q1 - q0) * (MHD / 4); it += blockDim.x) {
      const int qi = q0 + it / (MHD / 4), c = (it % (MHD / 4)) * 4;
      float mv[8], lv[8];
      float M = -INFINITY;
#pragma unroll
      for (int r = 0; r < 8; ++r) {
        mv[r] = -INFINITY;
        lv[r] = 0.f;
        if (r < S) {
          const uint32_t a = dsmem_addr(part_u32 + static_cast<uint32_t>((qi * PREC + MHD) * 4), r);
          mv[r] = ld_dsmem(a);
          lv[r] = ld_dsmem(a + 4);
          M = fmaxf(M, mv[r]);
        }
      }
      float L = 0.f;
      float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
      for (int r = 0; r < 8; ++r) {
        if (r < S) {
          const float w = (M == -INFINITY || mv[r] == -INFINITY) ? 0.f : expf(mv[r] - M);
          L += w * lv[r];
          const float4 v = ld_dsmem4(dsmem_addr(part_u32 + static_cast<uint32_t>((qi * PREC + c) * 4), r));
          acc.x += w * v.x; acc.y += w * v.y; acc.z += w * v.z; acc.w += w * v.w;
        }
      }
      const float inv = L > 0.f ? 1.f / L : 0.f;
      const size_t o_idx = static_cast<size_t>(b * p.q_rows + qi) * p.ldo + h * MHD + c;
      store_act(out, out_lo, o_idx, acc.x * inv);
      store_act(out, out_lo, o_idx + 1, acc.y * inv);
      store_act(out, out_lo, o_idx + 2, acc.z * inv);
      store_act(out, out_lo, o_idx + 3, acc.w * inv);
    }
  }
  cluster_sync();  // peers may still read this CTA's partials until here
  ATRACE(5);
}

template <bool SPLIT>
size_t tree_smem() {
  return TREE_STAGES * static_cast<size_t>(SPLIT ? 4 : 2) * MKT * MLDS * sizeof(bf16);
}

template <bool SPLIT>
cudaError_t launch_tree(const AttnParams& p, cudaStream_t s) {
  const size_t smem = tree_smem<SPLIT>();
  static bool attr = false;
  if (!attr) {
    cudaFuncSetAttribute(attn_tree_kernel<SPLIT>, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
    attr = true;
  }
  cudaLaunchAttribute at[2];
  int na = 0;
  at[na].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  at[na].val.programmaticStreamSerializationAllowed = 1;
  ++na;
  if (p.splits > 1) {
    at[na].id = cudaLaunchAttributeClusterDimension;
    at[na].val.clusterDim.x = p.splits;
    at[na].val.clusterDim.y = 1;
    at[na].val.clusterDim.z = 1;
    ++na;
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(p.splits, p.H, p.B);
  cfg.blockDim = dim3(MWARPS * 32);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cfg.attrs = at;
  cfg.numAttrs = na;
  cudaLaunchKernelEx(&cfg, attn_tree_kernel<SPLIT>, p);
  return cudaGetLastError();
}

// Largest cluster size <= want (and <= 8) whose B * H clusters are all resident at once.
template <bool SPLIT>
int tree_splits(int BH, int want) {
  static bool attr = false;
  if (!attr) {
    cudaFuncSetAttribute(attn_tree_kernel<SPLIT>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                         static_cast<int>(tree_smem<SPLIT>()));
    attr = true;
  }
  int S = std::max(1, std::min(8, want));
  for (; S > 1; --S) {
    cudaLaunchAttribute at[1];
    at[0].id = cudaLaunchAttributeClusterDimension;
    at[0].val.clusterDim.x = S;
    at[0].val.clusterDim.y = 1;
    at[0].val.clusterDim.z = 1;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(S, BH, 1);
    cfg.blockDim = dim3(MWARPS * 32);
    cfg.dynamicSmemBytes = tree_smem<SPLIT>();
    cfg.attrs = at;
    cfg.numAttrs = 1;
    int n = 0;
    if (cudaOccupancyMaxActiveClusters(&n, attn_tree_kernel<SPLIT>, &cfg) == cudaSuccess && n >= BH) break;
    cudaGetLastError();
  }
  return S;
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

bool attn_fuses_rope(int dtype, int hd) { return dtype == 1 && hd == 128; }

int attn_pick_splits(int dtype, int hd, int planes, int B, int H, int want) {
  if (!attn_fuses_rope(dtype, hd)) return want;
  return planes == 4 ? tree_splits<true>(B * H, want) : tree_splits<false>(B * H, want);
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
    return p.planes == 4 ? launch_tree<true>(p, s) : launch_tree<false>(p, s);
  } else if (p.hd == 64) {
    if (p.qkv) return cudaErrorInvalidValue;
    return launch<bf16, bf16, 64>(p, s);
  }
  return cudaErrorInvalidValue;
}

}  // namespace chimera
