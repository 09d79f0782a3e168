// Tree-masked attention on the 5th-generation tensor cores (bf16 models, head_dim 128).
//
// One CTA per (KV split s, head h, sequence b); the S splits of a (b, h) form one
// thread-block cluster and merge their partial states through distributed shared
// memory.  Per 64-key tile of the CTA's key range:
//
//   S  = Q K^T    tcgen05.mma, M = 64 queries, N = 64 keys, K = 128 dims, fp32 in TMEM
//   P  = exp(S - m) on the softmax warps (tcgen05.ld of S, mask, online max/sum)
//   O += P V      tcgen05.mma, M = 64 queries, N = 128 dims, K = 64 keys, fp32 in TMEM
//
// Every bf16 operand is a two-term split x = hi + lo of an fp32 value (queries, keys,
// values, probabilities); each product takes hi*hi + lo*hi + hi*lo, so the result
// matches fp32 arithmetic to ~2^-16.  Q, K and V tiles sit in shared memory in the
// K-major 128-byte-swizzled layout (V is read MN-major by the PV product); P is written
// by the softmax warps in the same layout.  Two S accumulators in tensor memory let the
// QK product of tile t+1 overlap the softmax of tile t.  The running max is only raised
// (and O rescaled) when a row's maximum grows by more than a factor ~e^8 (keeping P, l
// and O finite in fp32); the final normalisation uses the same max, so the result is
// exact.  Scores and maxima are kept in base-2 units (scaled by log2 e).
//
// Warps: 0..7 softmax + epilogue (warp w: tensor-memory lanes 32 (w % 4).., rows
// 16 (w % 4) .. + 15, keys / output columns of half w / 4), 8 loads the KV tiles (one thread issues TMA copies of 16-row page boxes into
// two-stage rings for K and for V, 128-byte swizzle applied by the copy engine), 9
// issues the MMAs and owns the tensor-memory allocation.
#include <algorithm>
#include <cmath>
#include <cstring>
#include <mutex>

#include "common.cuh"
#include "kernels.h"

namespace chimera {
namespace {

constexpr int HD = 128;
constexpr int KT = 64;                      // keys per tile
constexpr int NQ = 64;                      // query rows (UMMA M)
constexpr int SOFT_WARPS = 8, LOAD_WARPS = 1;  // softmax: warps w and w + 4 share rows, split keys
constexpr int THREADS = (SOFT_WARPS + LOAD_WARPS + 1) * 32;
constexpr int MMA_WARP = SOFT_WARPS + LOAD_WARPS;
constexpr int ATOM_ROWS64 = 64 * 128;       // bytes of one 64-row x 128-byte swizzle atom column
constexpr int TILE64 = 2 * ATOM_ROWS64;     // 64 rows x 128 bf16 (two atoms): 16 KB
constexpr int STAGES = 2;
constexpr int L2_AHEAD = 3;                 // tiles requested into L2 beyond the newest ring load
constexpr int PAGE_CACHE = 1024;
constexpr float RESCALE_LOG2 = 11.5f;        // raise the running max when it grows by > 2^11.5 (~e^8)
constexpr uint32_t TMEM_COLS = 256;          // S[2] (64 cols each) + O (128 cols)
constexpr int PREC = HD + 4;                 // partial record (o[128], m, l, pad)

// Byte offset of 16-byte chunk c (0..7) of row r inside a 128-byte-swizzled atom column.
__device__ __forceinline__ uint32_t swz(int r, int c) {
  return static_cast<uint32_t>((r >> 3) * 1024 + (r & 7) * 128 + ((c ^ (r & 7)) << 4));
}

// K-major (or, for the PV B operand, MN-major) 128-byte-swizzled smem descriptor.
__device__ __forceinline__ uint64_t desc_sw128(uint32_t addr, uint32_t lbo, uint32_t sbo) {
  uint64_t d = 0;
  d |= static_cast<uint64_t>((addr & 0x3FFFFu) >> 4);
  d |= static_cast<uint64_t>((lbo >> 4) & 0x3FFFu) << 16;
  d |= static_cast<uint64_t>((sbo >> 4) & 0x3FFFu) << 32;
  d |= static_cast<uint64_t>(1) << 46;
  d |= static_cast<uint64_t>(2) << 61;
  return d;
}

// kind::f16 instruction descriptor: D fp32, A and B bf16, A K-major, B K-major or
// MN-major (b_mn), shape M x N.
__device__ __forceinline__ uint32_t idesc_f16(int m, int n, bool b_mn) {
  return (1u << 4) | (1u << 7) | (1u << 10) | (b_mn ? (1u << 16) : 0u) | (static_cast<uint32_t>(n >> 3) << 17) |
         (static_cast<uint32_t>(m >> 4) << 24);
}

// 16x32bx2 access shape: lanes 0..15 of the warp read (write) TMEM lanes 0..15 of the
// warp's sub-partition at the addressed column, lanes 16..31 the same TMEM lanes at the
// column plus OFS; each of the 16 registers is the next column.
template <int OFS>
__device__ __forceinline__ void tmem_ld16x2(uint32_t taddr, uint32_t* r) {
  asm volatile(
      "tcgen05.ld.sync.aligned.16x32bx2.x16.b32 "
      "{%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15}, [%16], %17;"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
      : "r"(taddr), "n"(OFS));
}
template <int OFS>
__device__ __forceinline__ void tmem_st16x2(uint32_t taddr, const uint32_t* r) {
  asm volatile(
      "tcgen05.st.sync.aligned.16x32bx2.x16.b32 [%0], %1, "
      "{%2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, %16, %17};" ::"r"(taddr), "n"(OFS), "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]), "r"(r[8]), "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]), "r"(r[15])
      : "memory");
}
// Wait for the issued TMEM loads; the registers are operands so that no use of them is
// scheduled before the wait.
__device__ __forceinline__ void tmem_wait_ld16(uint32_t (&r)[16]) {
  asm volatile("tcgen05.wait::ld.sync.aligned;"
               : "+r"(r[0]), "+r"(r[1]), "+r"(r[2]), "+r"(r[3]), "+r"(r[4]), "+r"(r[5]), "+r"(r[6]), "+r"(r[7]), "+r"(r[8]), "+r"(r[9]), "+r"(r[10]), "+r"(r[11]), "+r"(r[12]), "+r"(r[13]), "+r"(r[14]), "+r"(r[15])
               :
               : "memory");
}
__device__ __forceinline__ void tmem_wait_ld32(uint32_t (&r)[32]) {
  asm volatile("tcgen05.wait::ld.sync.aligned;"
               : "+r"(r[0]), "+r"(r[1]), "+r"(r[2]), "+r"(r[3]), "+r"(r[4]), "+r"(r[5]), "+r"(r[6]), "+r"(r[7]), "+r"(r[8]), "+r"(r[9]), "+r"(r[10]), "+r"(r[11]), "+r"(r[12]), "+r"(r[13]), "+r"(r[14]), "+r"(r[15]), "+r"(r[16]), "+r"(r[17]), "+r"(r[18]), "+r"(r[19]), "+r"(r[20]), "+r"(r[21]), "+r"(r[22]), "+r"(r[23]), "+r"(r[24]), "+r"(r[25]), "+r"(r[26]), "+r"(r[27]), "+r"(r[28]), "+r"(r[29]), "+r"(r[30]), "+r"(r[31])
               :
               : "memory");
}
// 2^x on the special-function unit (inputs here are <= 0; results below 2^-126 flush to 0)
__device__ __forceinline__ float ex2_approx(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}
__device__ __forceinline__ void tmem_wait_st() { asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory"); }
__device__ __forceinline__ void fence_async_smem() { asm volatile("fence.proxy.async.shared::cta;" ::: "memory"); }

__device__ __forceinline__ void fence_async_global() { asm volatile("fence.proxy.async.global;" ::: "memory"); }

// Kernel arguments: the tensor map of the pool viewed as [pool_rows][hd] bf16 (box
// 64 dims x 16 rows) and the attention parameters.
struct TcArgs {
  CUtensorMap kv_map;
  AttnParams p;
};

__device__ __forceinline__ uint32_t pack_bf16x2(float a, float b) {
  const __nv_bfloat162 v = __floats2bfloat162_rn(a, b);
  return *reinterpret_cast<const uint32_t*>(&v);
}
// (a, b) -> hi pair, lo pair (lo = rounding residual of hi)
__device__ __forceinline__ void split_pair(float a, float b, uint32_t& hi, uint32_t& lo) {
  const __nv_bfloat162 h = __floats2bfloat162_rn(a, b);
  const float2 hf = __bfloat1622float2(h);
  hi = *reinterpret_cast<const uint32_t*>(&h);
  lo = pack_bf16x2(a - hf.x, b - hf.y);
}

// Two-term bf16 split of four values: hi (4 x bf16) and lo = the rounding residual.
__device__ __forceinline__ void split4(float4 v, uint2& hi, uint2& lo) {
  split_pair(v.x, v.y, hi.x, lo.x);
  split_pair(v.z, v.w, hi.y, lo.y);
}

// Under the M = 64 data-path layout, query rows 16q .. 16q + 15 sit in TMEM lanes 0..15 of
// sub-partition q (warp w reaches sub-partition w % 4).


template <bool SPLIT>
__global__ void __launch_bounds__(THREADS, 1) attn_tc_kernel(const __grid_constant__ TcArgs args) {
  const AttnParams& p = args.p;
  constexpr int NP = SPLIT ? 4 : 2;
  constexpr int KP = NP / 2;                 // planes of K (and of V): hi (, lo)
  constexpr int HALF_BYTES = KP * TILE64;   // one stage of K or of V
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  uint8_t* q_hi = smem;                     // 64 x 128 (two atoms)
  uint8_t* q_lo = q_hi + TILE64;
  uint8_t* p_buf = q_lo + TILE64;           // [2 buffers][hi, lo] 64 x 64 (one atom each, 8 KB)
  uint8_t* kbuf = p_buf + 4 * (NQ * 128);   // [STAGES][KP planes] 64 keys x 128 dims
  uint8_t* vbuf = kbuf + STAGES * HALF_BYTES;
  float* part = reinterpret_cast<float*>(kbuf);  // [64][PREC], reuses the KV stages after the loop
  uint64_t* bars = reinterpret_cast<uint64_t*>(vbuf + STAGES * HALF_BYTES);
  uint64_t* k_full = bars;           // [2] count 1 + transaction bytes (TMA)
  uint64_t* v_full = bars + 2;       // [2] count 1 + transaction bytes (TMA)
  uint64_t* k_empty = bars + 4;      // [2] tcgen05.commit after QK
  uint64_t* v_empty = bars + 6;      // [2] tcgen05.commit after PV
  uint64_t* s_full = bars + 8;       // [2] tcgen05.commit
  uint64_t* s_free = bars + 10;      // [2] count 4 (softmax warps)
  uint64_t* p_full = bars + 12;      // [2] count 4
  uint64_t* pv_done = bars + 14;     // [2] tcgen05.commit
  uint64_t* o_done = bars + 16;      // tcgen05.commit
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 17);
  int* s_abort = reinterpret_cast<int*>(tmem_slot + 1);
  int* s_pages = s_abort + 2;        // [PAGE_CACHE]
  float* s_stat = reinterpret_cast<float*>(s_pages + PAGE_CACHE);  // [64][2] final (m, l)
  float* s_xm = s_stat + 2 * NQ;     // [2 tiles][2 halves][64] tile maxima of the key halves
  float* s_lh = s_xm + 4 * NQ;       // [2 halves][64] partial row sums
  volatile int* abort = s_abort;

  const int s = blockIdx.x, h = blockIdx.y, b = blockIdx.z;
  const int S = gridDim.x;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  bf16* pool = static_cast<bf16*>(const_cast<void*>(p.pool)) + static_cast<size_t>(p.layer) * p.pool_layer_stride;

  if (threadIdx.x == 0) {
    for (int i = 0; i < 2; ++i) {
      mbar_init(&k_full[i], 1);
      mbar_init(&v_full[i], 1);
      mbar_init(&k_empty[i], 1);
      mbar_init(&v_empty[i], 1);
      mbar_init(&s_full[i], 1);
      mbar_init(&s_free[i], SOFT_WARPS);
      mbar_init(&p_full[i], SOFT_WARPS);
      mbar_init(&pv_done[i], 1);
    }
    mbar_init(o_done, 1);
    *s_abort = 0;
    mbar_fence_init();
  }
  if (warp == MMA_WARP) tmem_alloc(tmem_slot, TMEM_COLS);

  if (!p.prewait_kv) pdl_wait();
  const int nctx = p.n_ctx[b];
  // Local mode (fused projections, local rows starting at row 0: verify, prefill, plain
  // decoding, the draft's first sub-step): every local row is written by this launch,
  // so the local rows form one extra tile that the CTA owning it builds in shared
  // memory from the projections (no round trip through the pool); the committed rows
  // are tiles of the pool.  The local tile is the last of the split's virtual tiles
  // (so it goes to the CTA with the fewest committed tiles) and that CTA's first tile
  // (stage 0, free at start).  Otherwise the tiles cover slots [0, nctx + n_local).
  const bool lmode = p.qkv != nullptr && p.q_local0 == 0;
  const int ntiles = lmode ? (nctx + KT - 1) / KT : (nctx + p.n_local + KT - 1) / KT;  // tiles of the pool
  const int T = ntiles + (lmode ? 1 : 0);
  const int tps = (T + S - 1) / S;
  const int v0 = min(T, s * tps), v1 = min(T, v0 + tps);
  const int hl = (lmode && v0 < v1 && v1 == T) ? 1 : 0;  // this CTA holds the local tile (index 0)
  const int t0 = v0;                                    // pool tiles [t0, t1), tile indices hl ..
  const int t1 = hl ? T - 1 : v1;
  const int nt = hl + (t1 - t0);
  const bool cached = (t1 - t0) * 4 <= PAGE_CACHE;
  if (cached) {
    const int np = min((t1 - t0) * 4, p.max_pages - t0 * 4);
    for (int i = threadIdx.x; i < np; i += blockDim.x) s_pages[i] = p.page_table[b * p.max_pages + t0 * 4 + i];
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  // ---- KV staging (the loader warp, all lanes together): K or V of tile t into stage st
  // as 4 pages x KP planes x 2 swizzle atoms of 16 rows, one box per lane; pages at or
  // past kend are requested out of bounds (zero fill). One thread issues a box only every
  // ~70 ns, so the 8 KP boxes of a half go out from as many lanes at once. ----
  const long long rows_per_layer = p.pool_layer_stride / HD;
  auto issue_half = [&](int t, int st, int kend, bool is_v) {
    uint64_t* bar = is_v ? &v_full[st] : &k_full[st];
    if (lane == 0) mbar_arrive_expect_tx(bar, static_cast<uint32_t>(HALF_BYTES));
    __syncwarp();
    if (lane < 8 * KP) {
      const int u = lane / (2 * KP), plane = (lane >> 1) % KP, a = lane & 1;
      const int kg = t * KT + u * 16;
      long long y = p.pool_rows;  // out of bounds
      if (kg < kend) {
        const int page = cached ? s_pages[(t - t0) * 4 + u] : p.page_table[b * p.max_pages + t * 4 + u];
        y = static_cast<long long>(p.layer) * rows_per_layer +
            ((static_cast<long long>(page) * p.H + h) * NP + (is_v ? KP : 0) + plane) * 16;
      }
      uint8_t* base = (is_v ? vbuf : kbuf) + st * HALF_BYTES;
      tma_load_2d(base + plane * TILE64 + a * ATOM_ROWS64 + u * 16 * 128, &args.kv_map, a * 64,
                  static_cast<int>(y), bar);
    }
  };

  // L2 prefetch of tile t's page-planes (NP x 4 KB, contiguous per page), one page per lane
  auto prefetch_tile = [&](int t, int kend) {
    if (lane < 4 && t * KT + lane * 16 < kend) {
      const int page = cached ? s_pages[(t - t0) * 4 + lane] : p.page_table[b * p.max_pages + t * 4 + lane];
      const bf16* src = pool + (static_cast<size_t>(page) * p.H + h) * NP * 16 * HD;
      prefetch_l2_bulk(src, NP * 16 * HD * 2);
    }
  };
  int pf = 0;  // tiles [0, pf) of the range were requested into L2

  int pre = 0;  // leading tiles (K and V) requested before the dependency wait
  if (p.prewait_kv) {
    if (warp == SOFT_WARPS) {
      if (lane == 0) prefetch_tensormap(&args.kv_map);
      __syncwarp();
      // pool tiles whose rows are all committed (local mode: rows at or past nctx are
      // masked; the pool holds finite values there, the pools being cleared at set-up)
      while (hl + pre < nt && hl + pre < STAGES && (lmode || (t0 + pre + 1) * KT <= nctx)) {
        issue_half(t0 + pre, (hl + pre) & 1, nctx, false);
        issue_half(t0 + pre, (hl + pre) & 1, nctx, true);
        ++pre;
      }
      for (; pf < t1 - t0 && pf < STAGES + L2_AHEAD && (lmode || (t0 + pf + 1) * KT <= nctx); ++pf)
        if (pf >= pre) prefetch_tile(t0 + pf, nctx);
    }
    pdl_wait();
  }
  pdl_trigger();

  const int nloc = min(p.n_local_dev ? p.n_local_dev[b] : p.n_local, p.n_local);
  const int nq = p.nq_dev ? p.nq_dev[b] : p.nq;
  const int total = nctx + nloc;
  const int dm = p.H * HD;

  // ---- queries: rotate (fused mode), split, write the swizzled Q tiles ----
  for (int it = threadIdx.x; it < NQ * 8; it += blockDim.x) {
    const int r = it >> 3, j = it & 7;  // row, 8-dim chunk j of the first half (dims 8j.., 64 + 8j..)
    float lo_half[8], hi_half[8];
    if (r < nq) {
      const float* src = p.qkv ? p.qkv + static_cast<size_t>(b * p.q_rows + r) * p.ldqkv + h * HD + 8 * j
                               : p.q + static_cast<size_t>(b * p.q_rows + r) * p.ldq + h * HD + 8 * j;
      const float4 a0 = *reinterpret_cast<const float4*>(src), a1 = *reinterpret_cast<const float4*>(src + 4);
      const float4 b0 = *reinterpret_cast<const float4*>(src + HD / 2),
                   b1 = *reinterpret_cast<const float4*>(src + HD / 2 + 4);
      const float x1[8] = {a0.x, a0.y, a0.z, a0.w, a1.x, a1.y, a1.z, a1.w};
      const float x2[8] = {b0.x, b0.y, b0.z, b0.w, b1.x, b1.y, b1.z, b1.w};
      if (p.qkv) {
        const int pos = min(max(nctx + p.pos_base + (p.pos_off ? p.pos_off[r] : r), 0), p.max_pos - 1);
        const float2* tab = p.rope + static_cast<size_t>(pos) * (HD / 2) + 8 * j;
#pragma unroll
        for (int e = 0; e < 8; ++e) {
          const float2 cs = tab[e];
          lo_half[e] = x1[e] * cs.x - x2[e] * cs.y;
          hi_half[e] = x2[e] * cs.x + x1[e] * cs.y;
        }
      } else {
#pragma unroll
        for (int e = 0; e < 8; ++e) {
          lo_half[e] = x1[e];
          hi_half[e] = x2[e];
        }
      }
    } else {
#pragma unroll
      for (int e = 0; e < 8; ++e) lo_half[e] = hi_half[e] = 0.f;
    }
    uint4 h0, l0, h1, l1;
    split_pair(lo_half[0], lo_half[1], h0.x, l0.x);
    split_pair(lo_half[2], lo_half[3], h0.y, l0.y);
    split_pair(lo_half[4], lo_half[5], h0.z, l0.z);
    split_pair(lo_half[6], lo_half[7], h0.w, l0.w);
    split_pair(hi_half[0], hi_half[1], h1.x, l1.x);
    split_pair(hi_half[2], hi_half[3], h1.y, l1.y);
    split_pair(hi_half[4], hi_half[5], h1.z, l1.z);
    split_pair(hi_half[6], hi_half[7], h1.w, l1.w);
    *reinterpret_cast<uint4*>(q_hi + swz(r, j)) = h0;
    *reinterpret_cast<uint4*>(q_lo + swz(r, j)) = l0;
    *reinterpret_cast<uint4*>(q_hi + ATOM_ROWS64 + swz(r, j)) = h1;
    *reinterpret_cast<uint4*>(q_lo + ATOM_ROWS64 + swz(r, j)) = l1;
  }
  // the P tiles' rows are all rewritten every tile; nothing else to clear

  // ---- local mode: the owner of the local tile rotates k, writes k and v of the fresh
  // rows to the pool (for later steps) and into its stage-0 K and V tiles; rows past the
  // fresh ones are zero there ----
  if (hl) {
    for (int it = threadIdx.x; it < KT * 16; it += blockDim.x) {
      const int i = it >> 4, j = (it & 15) * 4;  // local row, pair index j .. j + 3 of the first half
      uint2 kh0 = make_uint2(0u, 0u), kl0 = kh0, kh1 = kh0, kl1 = kh0, vh0 = kh0, vl0 = kh0, vh1 = kh0, vl1 = kh0;
      if (i < nq) {
        const int slot = nctx + i;
        const int pos = nctx + p.pos_base + (p.pos_off ? p.pos_off[i] : i);
        if (pos < 0 || pos >= p.max_pos || (slot >> 4) >= p.max_pages) {
          if (p.err) atomicOr(p.err, ERR_CAPACITY);
        } else {
          const float* src = p.qkv + static_cast<size_t>(b * p.q_rows + i) * p.ldqkv + h * HD + j;
          const float4 k1 = *reinterpret_cast<const float4*>(src + dm);
          const float4 k2 = *reinterpret_cast<const float4*>(src + dm + HD / 2);
          const float4 v1 = *reinterpret_cast<const float4*>(src + 2 * dm);
          const float4 v2 = *reinterpret_cast<const float4*>(src + 2 * dm + HD / 2);
          const float2* tab = p.rope + static_cast<size_t>(pos) * (HD / 2) + j;
          const float4 cs01 = *reinterpret_cast<const float4*>(tab);
          const float4 cs23 = *reinterpret_cast<const float4*>(tab + 2);
          const float4 c = make_float4(cs01.x, cs01.z, cs23.x, cs23.z);
          const float4 sn = make_float4(cs01.y, cs01.w, cs23.y, cs23.w);
          split4(rot_lo(k1, k2, c, sn), kh0, kl0);
          split4(rot_hi(k1, k2, c, sn), kh1, kl1);
          split4(v1, vh0, vl0);
          split4(v2, vh1, vl1);
          const int page = p.page_table[b * p.max_pages + (slot >> 4)];
          bf16* base = pool + (static_cast<size_t>(page) * p.H + h) * NP * 16 * HD + (slot & 15) * HD + j;
          constexpr size_t plane = 16 * HD;
          if (SPLIT) {
            *reinterpret_cast<uint2*>(base) = kh0;
            *reinterpret_cast<uint2*>(base + plane) = kl0;
            *reinterpret_cast<uint2*>(base + HD / 2) = kh1;
            *reinterpret_cast<uint2*>(base + plane + HD / 2) = kl1;
            *reinterpret_cast<uint2*>(base + 2 * plane) = vh0;
            *reinterpret_cast<uint2*>(base + 3 * plane) = vl0;
            *reinterpret_cast<uint2*>(base + 2 * plane + HD / 2) = vh1;
            *reinterpret_cast<uint2*>(base + 3 * plane + HD / 2) = vl1;
          } else {
            *reinterpret_cast<uint2*>(base) = kh0;
            *reinterpret_cast<uint2*>(base + HD / 2) = kh1;
            *reinterpret_cast<uint2*>(base + plane) = vh0;
            *reinterpret_cast<uint2*>(base + plane + HD / 2) = vh1;
          }
        }
      }
      // stage 0: row i, dims j .. j + 3 (atom 0) and 64 + j .. (atom 1): half of chunk j / 8
      const uint32_t o0 = swz(i, j >> 3) + ((j & 7) << 1);
      const uint32_t o1 = ATOM_ROWS64 + o0;
      uint8_t* kt = kbuf;
      uint8_t* vt = vbuf;
      *reinterpret_cast<uint2*>(kt + o0) = kh0;
      *reinterpret_cast<uint2*>(kt + o1) = kh1;
      *reinterpret_cast<uint2*>(vt + o0) = vh0;
      *reinterpret_cast<uint2*>(vt + o1) = vh1;
      if (SPLIT) {
        *reinterpret_cast<uint2*>(kt + TILE64 + o0) = kl0;
        *reinterpret_cast<uint2*>(kt + TILE64 + o1) = kl1;
        *reinterpret_cast<uint2*>(vt + TILE64 + o0) = vl0;
        *reinterpret_cast<uint2*>(vt + TILE64 + o1) = vl1;
      }
    }
  }
  // ---- otherwise: fresh local rows of this CTA's key range: rotate k, write k and v to
  // the pool, read back by TMA ----
  if (p.qkv && !lmode) {
    const int fresh0 = nctx + p.q_local0;
    const int f0 = max(0, t0 * KT - fresh0), f1 = min(nq, t1 * KT - fresh0);
    for (int it = threadIdx.x; it < (f1 - f0) * 16; it += blockDim.x) {
      const int i = f0 + (it >> 4), j = (it & 15) * 4;
      const int slot = fresh0 + i;
      const int pos = nctx + p.pos_base + (p.pos_off ? p.pos_off[i] : i);
      if (pos < 0 || pos >= p.max_pos || (slot >> 4) >= p.max_pages) {
        if (p.err) atomicOr(p.err, ERR_CAPACITY);
        continue;
      }
      const int page = p.page_table[b * p.max_pages + (slot >> 4)];
      const float* src = p.qkv + static_cast<size_t>(b * p.q_rows + i) * p.ldqkv + h * HD + j;
      const float4 k1 = *reinterpret_cast<const float4*>(src + dm);
      const float4 k2 = *reinterpret_cast<const float4*>(src + dm + HD / 2);
      const float4 v1 = *reinterpret_cast<const float4*>(src + 2 * dm);
      const float4 v2 = *reinterpret_cast<const float4*>(src + 2 * dm + HD / 2);
      const float2* tab = p.rope + static_cast<size_t>(pos) * (HD / 2) + j;
      const float4 cs01 = *reinterpret_cast<const float4*>(tab);
      const float4 cs23 = *reinterpret_cast<const float4*>(tab + 2);
      const float4 c = make_float4(cs01.x, cs01.z, cs23.x, cs23.z);
      const float4 sn = make_float4(cs01.y, cs01.w, cs23.y, cs23.w);
      const float4 ka = rot_lo(k1, k2, c, sn), kb = rot_hi(k1, k2, c, sn);
      bf16* base = pool + (static_cast<size_t>(page) * p.H + h) * NP * 16 * HD + (slot & 15) * HD + j;
      constexpr size_t plane = 16 * HD;
      if (SPLIT) {
        store4_split(base, base + plane, ka);
        store4_split(base + HD / 2, base + plane + HD / 2, kb);
        store4_split(base + 2 * plane, base + 3 * plane, v1);
        store4_split(base + 2 * plane + HD / 2, base + 3 * plane + HD / 2, v2);
      } else {
        store4<bf16>(base, ka);
        store4<bf16>(base + HD / 2, kb);
        store4<bf16>(base + plane, v1);
        store4<bf16>(base + plane + HD / 2, v2);
      }
    }
    fence_async_global();  // the rows are read back by TMA (async proxy)
  }
  fence_async_smem();  // the Q tiles (and the local K, V tile) are read by the tensor cores (async proxy)
  __threadfence_block();
  __syncthreads();
  if (hl && threadIdx.x == 0) {  // the local tile is in place: stage 0 of K and V is full
    mbar_arrive(&k_full[0]);
    mbar_arrive(&v_full[0]);
  }

  if (warp == SOFT_WARPS) {
    // ---------------- KV loader (the whole warp; lane 0 polls and decides) ----------------
    if (!p.prewait_kv && lane == 0) prefetch_tensormap(&args.kv_map);
    __syncwarp();
    // K of tile j needs the QK product of tile j - 2 done, V of tile j the PV product
    // of tile j - 2; both are polled so that neither waits behind the other
    // tile index i: the local tile (i = 0 when hl) or pool tile t0 + i - hl, stage i & 1
    const int kend = lmode ? nctx : total;
    int nk = hl + pre, nv = hl + pre;
    uint64_t last_progress = global_timer_ns();
    while (nk < nt || nv < nt) {
      bool moved = false;
      const int kgo = __shfl_sync(0xffffffffu, (lane == 0 && nk < nt &&
                                                (nk < STAGES || mbar_test(&k_empty[nk & 1], ((nk - STAGES) >> 1) & 1))) ? 1 : 0, 0);
      if (kgo) {
        issue_half(t0 + nk - hl, nk & 1, kend, false);
        for (pf = max(pf, nk - hl + 1); pf < t1 - t0 && pf <= nk - hl + L2_AHEAD; ++pf) prefetch_tile(t0 + pf, kend);
        ++nk;
        moved = true;
      }
      const int vgo = __shfl_sync(0xffffffffu, (lane == 0 && nv < nk &&
                                                (nv < STAGES || mbar_test(&v_empty[nv & 1], ((nv - STAGES) >> 1) & 1))) ? 1 : 0, 0);
      if (vgo) {
        issue_half(t0 + nv - hl, nv & 1, kend, true);
        ++nv;
        moved = true;
      }
      int quit = 0;
      if (lane == 0) {
        if (moved)
          last_progress = global_timer_ns();
        else if (global_timer_ns() - last_progress > 2000000000ull)
          *abort = 1;
        quit = *abort;
      }
      if (__shfl_sync(0xffffffffu, quit, 0)) break;
    }
    // copies still in flight when the CTA gives up: let them land before it exits
    if (lane == 0 && *abort) {
      for (int j = nk - 1; j >= 0 && j >= nk - STAGES; --j) mbar_wait_plain(&k_full[j & 1], (j >> 1) & 1, 200000000ull);
      for (int j = nv - 1; j >= 0 && j >= nv - STAGES; --j) mbar_wait_plain(&v_full[j & 1], (j >> 1) & 1, 200000000ull);
    }
    __syncwarp();
  } else if (warp == MMA_WARP) {
    // ---------------- MMA issuer ----------------
    if (lane == 0 && nt > 0) {
      const uint32_t id_qk = idesc_f16(NQ, KT, false);
      const uint32_t id_pv = idesc_f16(NQ, HD, true);
      const uint32_t qh = smem_u32(q_hi), ql = smem_u32(q_lo);
      // descriptors are precomputed once; advancing a K-major operand by b bytes adds
      // b >> 4 to its start-address field (all operands lie below 256 KB of shared memory)
      const uint64_t dq_h = desc_sw128(qh, 16, 1024), dq_l = desc_sw128(ql, 16, 1024);
      uint64_t dk_h[STAGES], dv_h[STAGES], dp_h[2];
#pragma unroll
      for (int st = 0; st < STAGES; ++st) {
        dk_h[st] = desc_sw128(smem_u32(kbuf + st * HALF_BYTES), 16, 1024);
        // V as MN-major B: 64-dim atoms 8 KB apart (leading), 8-key groups 1 KB apart
        dv_h[st] = desc_sw128(smem_u32(vbuf + st * HALF_BYTES), ATOM_ROWS64, 1024);
      }
#pragma unroll
      for (int pb = 0; pb < 2; ++pb) dp_h[pb] = desc_sw128(smem_u32(p_buf + (2 * pb) * (NQ * 128)), 16, 1024);
      constexpr uint64_t LO_OFS = TILE64 >> 4;        // hi plane -> lo plane (16 KB)
      constexpr uint64_t P_LO_OFS = (NQ * 128) >> 4;  // P hi -> P lo (8 KB)
      auto pv = [&](int i) {  // O += P_i V_i
        const int st = i & 1;
        const uint32_t o_t = tmem + 128;
#pragma unroll
        for (int ks = 0; ks < KT / 16; ++ks) {
          const uint64_t a_h = dp_h[st] + static_cast<uint64_t>(ks * 2);  // 32 bytes per K step
          const uint64_t b_h = dv_h[st] + static_cast<uint64_t>(ks * 128);  // 16 keys = 2 KB
          tc_mma_bf16(o_t, a_h, b_h, id_pv, (i > 0 || ks > 0) ? 1u : 0u);
          tc_mma_bf16(o_t, a_h + P_LO_OFS, b_h, id_pv, 1u);
          if (SPLIT) tc_mma_bf16(o_t, a_h, b_h + LO_OFS, id_pv, 1u);
        }
        tc_commit(&pv_done[i & 1]);
        tc_commit(&v_empty[st]);
      };
      auto qk = [&](int i) {  // S_i = Q K_i^T into S buffer i & 1
        const int st = i & 1;
        const uint32_t s_t = tmem + st * 64;
#pragma unroll
        for (int ks = 0; ks < HD / 16; ++ks) {
          const uint64_t off = static_cast<uint64_t>(((ks >> 2) * ATOM_ROWS64 + (ks & 3) * 32) >> 4);
          const uint64_t b_h = dk_h[st] + off;
          tc_mma_bf16(s_t, dq_h + off, b_h, id_qk, ks > 0 ? 1u : 0u);
          tc_mma_bf16(s_t, dq_l + off, b_h, id_qk, 1u);
          if (SPLIT) tc_mma_bf16(s_t, dq_h + off, b_h + LO_OFS, id_qk, 1u);
        }
        tc_commit(&s_full[st]);
        tc_commit(&k_empty[st]);
      };
      // issue whichever product is ready: PV(np) when P and V of tile np are in, QK(nq)
      // when K is in, its S buffer is free and it runs at most one tile ahead of the PV
      // products (so no barrier is ever two phases ahead of its waiter)
      int nqk = 0, npv = 0;
      uint64_t last_progress = global_timer_ns();
      while (npv < nt && !*abort) {
        bool moved = false;
        if (npv < nqk && mbar_test(&p_full[npv & 1], (npv >> 1) & 1) &&
            mbar_test(&v_full[npv & 1], (npv >> 1) & 1)) {
          tc_fence_after();
          pv(npv);
          ++npv;
          moved = true;
        }
        if (nqk < nt && nqk <= npv + 1 && mbar_test(&k_full[nqk & 1], (nqk >> 1) & 1) &&
            (nqk < 2 || mbar_test(&s_free[nqk & 1], ((nqk - 2) >> 1) & 1))) {
          tc_fence_after();
          qk(nqk);
          ++nqk;
          moved = true;
        }
        if (moved) {
          last_progress = global_timer_ns();
        } else if (global_timer_ns() - last_progress > 2000000000ull) {
          *abort = 1;
        }
      }
      tc_commit(o_done);  // all MMAs issued by this thread, including any after an abort
      // tensor memory and the KV stages are released only after every MMA completed
      mbar_wait_plain(o_done, 0, 200000000ull);
    }
  } else {
    // ---------------- softmax (warps 0..7) ----------------
    // Warps w and w + 4 own the 16 rows of TMEM sub-partition w % 4 and the key halves
    // 0 / 1 of every tile; within a warp, lanes l and l + 16 share row l % 16 and take
    // 16 keys each (the 16x32bx2 access shape), so every lane works. The two lanes of a
    // row combine by a shuffle, the warp pair through shared memory (named barrier
    // 1 + w % 4). After a timeout the loop keeps running (without work) so both warps of
    // a pair still meet at every barrier.
    const int half = warp >> 2, quad = warp & 3, sub = lane >> 4;
    const int r = quad * 16 + (lane & 15);
    const bool live = r < nq;
    const int kofs = 32 * half + 16 * sub;  // this lane's first key within a tile
    const unsigned long long anc = live ? p.anc[p.q_local0 + r] : 0ull;
    const float scale2 = p.scale * 1.4426950408889634f;  // softmax in base 2: exp(x) = 2^(x log2 e)
    const uint32_t tlane = static_cast<uint32_t>(quad * 32) << 16;
    float m_used = -INFINITY, l = 0.f;
    bool dead = false;
    for (int i = 0; i < nt; ++i) {
      const int sb = i & 1;
      const bool loc = hl && i == 0;
      const int t = t0 + i - hl;
      bool ok = !dead && mbar_wait(&s_full[sb], (i >> 1) & 1, abort);
      dead = !__all_sync(0xffffffffu, ok);
      tc_fence_after();
      float sv[16];
      if (!dead) {
        uint32_t rr[16];
        tmem_ld16x2<16>(tmem + tlane + sb * 64 + half * 32, rr);
        tmem_wait_ld16(rr);
#pragma unroll
        for (int j = 0; j < 16; ++j) sv[j] = __uint_as_float(rr[j]);
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0 && !dead) mbar_arrive(&s_free[sb]);
      // visibility of this lane's 16 keys (bit j: key kofs + j of the tile): the local
      // tile's keys are local rows (ancestor mask), a pool tile's keys are slots 64 t ..
      uint32_t vbits = 0u;
      if (live) {
        unsigned long long vis;
        if (loc) {
          vis = anc & (nloc >= 64 ? ~0ull : ((1ull << nloc) - 1ull));
        } else {
          const int base = t * KT;
          const int nc = nctx - base, nv = total - base, off = base - nctx;
          const unsigned long long cm = nc >= 64 ? ~0ull : (nc <= 0 ? 0ull : ((1ull << nc) - 1ull));
          const unsigned long long lm =
              lmode ? 0ull : (off >= 0 ? (off < 64 ? (anc >> off) : 0ull) : (-off < 64 ? (anc << -off) : 0ull));
          const unsigned long long vm = nv >= 64 ? ~0ull : (nv <= 0 ? 0ull : ((1ull << nv) - 1ull));
          vis = (cm | lm) & vm;
        }
        vbits = static_cast<uint32_t>(vis >> kofs) & 0xFFFFu;
      }
      float ta = -INFINITY, tb = -INFINITY;  // two chains of maxima
#pragma unroll
      for (int j = 0; j < 16; ++j) {
        sv[j] = (!dead && ((vbits >> j) & 1u)) ? sv[j] * scale2 : -INFINITY;
        if (j & 1)
          tb = fmaxf(tb, sv[j]);
        else
          ta = fmaxf(ta, sv[j]);
      }
      // the row's maximum over its 64 keys: the other lane of the row, then the pair warp
      float tmax = fmaxf(ta, tb);
      tmax = fmaxf(tmax, __shfl_xor_sync(0xffffffffu, tmax, 16));
      if (sub == 0) s_xm[(sb * 2 + half) * NQ + r] = tmax;
      named_bar(1 + quad, 64);
      tmax = fmaxf(tmax, s_xm[(sb * 2 + (half ^ 1)) * NQ + r]);
      // this tile's P buffer was read by the PV product of tile i - 2
      if (i >= 2) {
        ok = !dead && mbar_wait(&pv_done[i & 1], ((i - 2) >> 1) & 1, abort);
        dead = !__all_sync(0xffffffffu, ok);
        tc_fence_after();
      }
      // m moves only when the tile's maximum exceeds it by more than 2^RESCALE_LOG2; O then
      // holds products of earlier tiles exactly when m was already finite. Both decisions
      // depend only on the row's shared maxima, so all four lanes of a row agree.
      const bool raise = tmax > m_used + RESCALE_LOG2 || (m_used == -INFINITY && tmax > -INFINITY);
      const bool rescale = raise && m_used != -INFINITY;
      float corr = 1.f;
      if (raise) {
        corr = rescale ? exp2f(m_used - tmax) : 0.f;
        m_used = tmax;
      }
      if (!dead && i > 0 && __any_sync(0xffffffffu, rescale)) {
        // O holds the products up to tile i - 1: wait for the last one before rescaling
        ok = mbar_wait(&pv_done[(i - 1) & 1], ((i - 1) >> 1) & 1, abort);
        dead = !__all_sync(0xffffffffu, ok);
        tc_fence_after();
        if (!dead) {
          // this warp's 64 columns of its O rows (lanes 0..15: the first 32, lanes
          // 16..31: the last 32); factor 1 for rows that kept m
          const float f = rescale ? corr : 1.f;
          const uint32_t oa = tmem + tlane + 128 + half * 64;
          uint32_t rr[32];
          tmem_ld16x2<32>(oa, rr);
          tmem_ld16x2<32>(oa + 16, rr + 16);
          tmem_wait_ld32(rr);
#pragma unroll
          for (int j = 0; j < 32; ++j) rr[j] = __float_as_uint(__uint_as_float(rr[j]) * f);
          tmem_st16x2<32>(oa, rr);
          tmem_st16x2<32>(oa + 16, rr + 16);
          tmem_wait_st();
        }
      }
      l *= corr;
      // P = 2^(S - m), two-term split into the swizzled P tile (this lane's 2 chunks)
      uint8_t* ph = p_buf + (2 * sb) * (NQ * 128);
      uint8_t* pl = ph + NQ * 128;
      float ra = 0.f, rb = 0.f;
#pragma unroll
      for (int c = 0; c < 2; ++c) {
        float pv8[8];
#pragma unroll
        for (int e = 0; e < 8; ++e) {
          const float x = sv[8 * c + e];
          pv8[e] = (x == -INFINITY) ? 0.f : ex2_approx(x - m_used);
          if (e & 1)
            rb += pv8[e];
          else
            ra += pv8[e];
        }
        uint4 hh, ll;
        split_pair(pv8[0], pv8[1], hh.x, ll.x);
        split_pair(pv8[2], pv8[3], hh.y, ll.y);
        split_pair(pv8[4], pv8[5], hh.z, ll.z);
        split_pair(pv8[6], pv8[7], hh.w, ll.w);
        if (!dead) {
          *reinterpret_cast<uint4*>(ph + swz(r, kofs / 8 + c)) = hh;
          *reinterpret_cast<uint4*>(pl + swz(r, kofs / 8 + c)) = ll;
        }
      }
      l += ra + rb;
      fence_async_smem();
      tc_fence_before();
      __syncwarp();
      if (lane == 0 && !dead) mbar_arrive(&p_full[sb]);
    }
    l += __shfl_xor_sync(0xffffffffu, l, 16);  // the row's sum over this warp's key half
    if (sub == 0) {
      if (half == 0) s_stat[2 * r] = m_used;
      s_lh[half * NQ + r] = l;
    }
  }

  // ---- epilogue: every CTA pushes its partial rows (O, m, l) to the cluster CTA that
  // finishes them (rows [r * ceil(nq / S), ...) belong to rank r); the receive buffer
  // reuses the KV rings, so the pushes start once every CTA of the cluster is past its
  // main loop (split cluster barrier) ----
  if (warp < SOFT_WARPS) {
    if (nt > 0) {
      mbar_wait(o_done, 0, abort);
      tc_fence_after();
    }
    __syncwarp();
  }
  __syncthreads();  // this CTA's rings are idle: every load landed and every MMA completed
  __syncwarp();
  if (S > 1) cluster_arrive();
  const int rpc = (nq + S - 1) / S;
  float* recv = part;                     // [S][rpc][PREC], S * rpc <= NQ + 7 rows (37.5 KB)
  float* s_w = part + (NQ + 8) * PREC;    // [rpc][8] merge weights, past the receive slots
  {
    const bool soft = warp < SOFT_WARPS;
    const int half = (warp >> 2) & 1, sub = lane >> 4;
    const int r = (warp & 3) * 16 + (lane & 15);
    const bool have = soft && nt > 0 && !*abort;
    const bool mine = soft && r < nq;
    const int cb = half * 64 + sub * 32;  // this lane's first O column
    uint32_t rr[32];
    if (have) {  // this lane's 32 columns of the O row, while the peers finish
      const uint32_t oa = tmem + (static_cast<uint32_t>((warp & 3) * 32) << 16) + 128 + half * 64;
      tmem_ld16x2<32>(oa, rr);
      tmem_ld16x2<32>(oa + 16, rr + 16);
      tmem_wait_ld32(rr);
    }
    __syncwarp();
    if (S > 1) cluster_wait();
    if (soft) {
      const int owner = mine ? r / rpc : 0;
      const uint32_t slot = smem_u32(recv + (s * rpc + (mine ? r - owner * rpc : 0)) * PREC);
      const uint32_t dst = S > 1 ? dsmem_addr(slot, owner) : slot;
      const float lr = mine ? s_lh[r] + s_lh[NQ + r] : 0.f;
      const bool keep = have && lr > 0.f;
      if (mine) {
#pragma unroll
        for (int j = 0; j < 32; j += 4) {
          const float4 v = keep ? make_float4(__uint_as_float(rr[j]), __uint_as_float(rr[j + 1]),
                                              __uint_as_float(rr[j + 2]), __uint_as_float(rr[j + 3]))
                                : make_float4(0.f, 0.f, 0.f, 0.f);
          st_dsmem4(dst + static_cast<uint32_t>((cb + j) * 4), v);
        }
        if (half == 0 && sub == 0) {
          st_dsmem(dst + HD * 4, nt > 0 ? s_stat[2 * r] : -INFINITY);
          st_dsmem(dst + (HD + 1) * 4, nt > 0 ? lr : 0.f);
        }
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  __syncwarp();
  if (warp == MMA_WARP) {
    tc_fence_after();
    tmem_dealloc(tmem, TMEM_COLS);
  }
  if (threadIdx.x == 0 && *abort && p.err) atomicOr(p.err, ERR_TIMEOUT);
  __syncwarp();
  if (S > 1) cluster_sync();  // every push into this CTA is complete and visible

  // ---- merge the S partials of this CTA's rows (local shared memory) ----
  bf16* out = static_cast<bf16*>(p.out);
  bf16* out_lo = static_cast<bf16*>(p.out_lo);
  const int q0 = s * rpc, nrows = max(0, min(nq, q0 + rpc) - q0);
  for (int rl = threadIdx.x; rl < nrows; rl += blockDim.x) {
    float mv[8], M = -INFINITY;
#pragma unroll
    for (int k = 0; k < 8; ++k) {
      mv[k] = k < S ? recv[(k * rpc + rl) * PREC + HD] : -INFINITY;
      M = fmaxf(M, mv[k]);
    }
    float L = 0.f;
#pragma unroll
    for (int k = 0; k < 8; ++k) {
      mv[k] = (k < S && M != -INFINITY && mv[k] != -INFINITY) ? exp2f(mv[k] - M) : 0.f;
      if (k < S) L += mv[k] * recv[(k * rpc + rl) * PREC + HD + 1];
    }
    const float inv = L > 0.f ? 1.f / L : 0.f;
#pragma unroll
    for (int k = 0; k < 8; ++k)
      if (k < S) s_w[rl * 8 + k] = mv[k] * inv;
  }
  __syncthreads();
  for (int it = threadIdx.x; it < nrows * (HD / 4); it += blockDim.x) {
    const int rl = it / (HD / 4), c = (it % (HD / 4)) * 4;
    float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
    for (int k = 0; k < 8; ++k) {
      if (k < S) {
        const float w = s_w[rl * 8 + k];
        const float4 v = *reinterpret_cast<const float4*>(recv + (k * rpc + rl) * PREC + c);
        acc.x += w * v.x; acc.y += w * v.y; acc.z += w * v.z; acc.w += w * v.w;
      }
    }
    const size_t o_idx = static_cast<size_t>(b * p.q_rows + q0 + rl) * p.ldo + h * HD + c;
    store_act4(out, out_lo, o_idx, acc);
  }
}

template <bool SPLIT>
size_t tc_smem() {
  const size_t np = SPLIT ? 4 : 2;
  return 1024 + 2 * TILE64 + 4 * NQ * 128 + STAGES * np * TILE64 + 18 * 8 + 16 + PAGE_CACHE * 4 + 8 * NQ * 4;
}

// The dynamic shared memory limit is an attribute of the device that is current when it
// is set: raised once per device (and kernel variant), the return code checked.
constexpr int ATT_MAX_DEVICES = 64;
std::mutex g_att_attr_mu;
bool g_att_attr[2][ATT_MAX_DEVICES];

template <bool SPLIT>
cudaError_t tc_attr() {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= ATT_MAX_DEVICES) return cudaErrorInvalidDevice;
  std::lock_guard<std::mutex> lk(g_att_attr_mu);
  if (!g_att_attr[SPLIT ? 1 : 0][dev]) {
    e = cudaFuncSetAttribute(attn_tc_kernel<SPLIT>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             static_cast<int>(tc_smem<SPLIT>()));
    if (e != cudaSuccess) return e;
    g_att_attr[SPLIT ? 1 : 0][dev] = true;
  }
  return cudaSuccess;
}

template <bool SPLIT>
cudaError_t launch_tc(const AttnParams& p, cudaStream_t s) {
  cudaError_t ae = tc_attr<SPLIT>();
  if (ae != cudaSuccess) return ae;
  TcArgs args;
  memset(&args, 0, sizeof(args));
  args.p = p;
  if (encode_2d_bf16(&args.kv_map, p.pool, HD, static_cast<uint64_t>(p.pool_rows), HD, 64, 16) != 0)
    return cudaErrorInvalidValue;
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
  cfg.blockDim = dim3(THREADS);
  cfg.dynamicSmemBytes = tc_smem<SPLIT>();
  cfg.stream = s;
  cfg.attrs = at;
  cfg.numAttrs = na;
  cudaLaunchKernelEx(&cfg, attn_tc_kernel<SPLIT>, args);
  return cudaGetLastError();
}

template <bool SPLIT>
int tc_splits(int BH, int want) {
  if (tc_attr<SPLIT>() != cudaSuccess) return 1;
  int S = std::max(1, std::min(8, want));
  for (; S > 1; --S) {
    cudaLaunchAttribute at[1];
    at[0].id = cudaLaunchAttributeClusterDimension;
    at[0].val.clusterDim.x = S;
    at[0].val.clusterDim.y = 1;
    at[0].val.clusterDim.z = 1;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(S, BH, 1);
    cfg.blockDim = dim3(THREADS);
    cfg.dynamicSmemBytes = tc_smem<SPLIT>();
    cfg.attrs = at;
    cfg.numAttrs = 1;
    int n = 0;
    if (cudaOccupancyMaxActiveClusters(&n, attn_tc_kernel<SPLIT>, &cfg) == cudaSuccess && n >= BH) break;
    cudaGetLastError();
  }
  return S;
}

}  // namespace


cudaError_t attention_tc(const AttnParams& p, cudaStream_t s) {
  if (p.hd != HD || p.nq_max > NQ || p.n_local > 64 || p.splits < 1 || p.splits > 8) return cudaErrorInvalidValue;
  // the TMA row coordinate is a 32-bit integer; the pool base must be 16-byte aligned
  if (p.pool_rows < 16 || p.pool_rows >= (1ll << 31) || (reinterpret_cast<uintptr_t>(p.pool) & 15))
    return cudaErrorInvalidValue;
  if (p.planes != 2 && p.planes != 4) return cudaErrorInvalidValue;
  if (p.qkv && (!p.rope || !p.err || p.max_pos < 1 || (p.ldqkv & 3))) return cudaErrorInvalidValue;
  if (!p.qkv && (p.ldq & 3)) return cudaErrorInvalidValue;
  return p.planes == 4 ? launch_tc<true>(p, s) : launch_tc<false>(p, s);
}

int attention_tc_splits(int planes, int BH, int want) {
  return planes == 4 ? tc_splits<true>(BH, want) : tc_splits<false>(BH, want);
}

}  // namespace chimera
