// Weight-streaming bf16 linear on the 5th-generation tensor cores (sm_103a).
//
//   Y[M][N] (epilogue)= X[M][K] . W[N][K]^T,  fp32 accumulation in tensor memory.
//
// Swap-AB: the weight tile (128 output features x 64 K) is the MMA's A operand
// (UMMA M = 128) and the token tile (BN rows x 64 K, BN = 16..256) is its B operand,
// so the skinny token dimension of the draft (1..8 rows) and of the tree verify
// (16..256 rows) becomes the MMA N.  At these sizes the kernel is bound by streaming
// W from HBM once.
//
// Work split: stream-K.  The (feature tile, token tile, K block) units are cut into
// gridDim.x equal contiguous ranges (one persistent CTA per SM), so every SM streams
// the same number of weight bytes whatever the matrix shape.  A tile whose K range
// spans several CTAs is finished by the last CTA to arrive (an atomic counter per
// tile): every contributor writes its fp32 partial to a workspace slot, and the last
// one sums the partials in contributor order (deterministic) and runs the epilogue.
// No CTA ever waits on another.
//
// Roles (192 threads): warp 0 issues TMA loads into an n-stage shared-memory ring,
// warp 1 issues tcgen05.mma into one of two TMEM accumulators, warps 2..5 drain the
// other accumulator (tcgen05.ld) and run the epilogue, so the loads of the next
// segment overlap the epilogue of the previous one.
#include <cstdio>
#include <cstring>
#include <atomic>
#include <mutex>

#include "common.cuh"
#include "launch.cuh"
#include "kernels.h"

namespace chimera {
namespace {

// Pipeline shape (compile-time; the defaults are the tuned values).
#ifndef CHIMERA_LIN_CTAS_PER_SM
#define CHIMERA_LIN_CTAS_PER_SM 1
#endif
#ifndef CHIMERA_LIN_PIPE_KB
#define CHIMERA_LIN_PIPE_KB 200
#endif
#ifndef CHIMERA_LIN_PRE_STAGES
#define CHIMERA_LIN_PRE_STAGES 2
#endif
#ifndef CHIMERA_LIN_BK_ATOMS
#define CHIMERA_LIN_BK_ATOMS 2
#endif
constexpr int BM = 128;   // weight rows per tile (UMMA M)
constexpr int ATOM = 64;  // one 128-byte swizzle atom of bf16 along K
constexpr int BKA = CHIMERA_LIN_BK_ATOMS;  // atoms per pipeline stage
constexpr int BK = ATOM * BKA;             // K per stage
constexpr int UK = 16;    // UMMA K for 16-bit inputs
constexpr int MAX_STAGES = 12;
constexpr int THREADS = 192;
constexpr int CTAS_PER_SM = CHIMERA_LIN_CTAS_PER_SM;
constexpr int PIPE_SMEM = CHIMERA_LIN_PIPE_KB * 1024;
constexpr int MAX_BN = 256;
constexpr int MAX_TILES = 8192;


// Stream-K partition in 32-bit arithmetic (the host checks units * grid < 2^32).
__device__ __forceinline__ int cta_of_unit(uint32_t u, uint32_t U, uint32_t G) {
  return static_cast<int>(((u + 1) * G - 1) / U);
}
__device__ __forceinline__ uint32_t unit_begin(uint32_t c, uint32_t U, uint32_t G) { return c * U / G; }

// Epilogue of 16 consecutive token columns (m0 .. m0+15) of feature row f.  All
// loads are issued before the stores so they overlap.
__device__ __forceinline__ void epi_store16(const TcLinearParams& p, int m0, int f, const float (&v)[16]) {
  if (f >= p.N) return;
  if (p.epi == EPI_RESID) {
    float* y = static_cast<float*>(p.Y);
#pragma unroll
    for (int j = 0; j < 16; ++j)
      if (m0 + j < p.M) red_add_f32(y + static_cast<size_t>(m0 + j) * p.ldy + f, v[j]);
    return;
  }
#pragma unroll
  for (int j = 0; j < 16; ++j) {
    if (m0 + j >= p.M) break;
    const float x = (p.epi == EPI_SILU) ? silu_f(v[j]) : v[j];
    const size_t idx = static_cast<size_t>(m0 + j) * p.ldy + f;
    if (p.out_f32)
      static_cast<float*>(p.Y)[idx] = x;
    else
      store_act(static_cast<bf16*>(p.Y), static_cast<bf16*>(p.Y2), idx, x);
  }
}

// EPI_RESID with float4 reductions: the warp's 32 feature rows x 16 token columns go
// through shared memory (sw: [16][33] floats) so that each lane adds runs of four
// consecutive features of one token (one vector red.global.add instead of four).
__device__ __forceinline__ void epi_red16(const TcLinearParams& p, int m0, int f0, int lane, const float (&v)[16],
                                          float* sw) {
#pragma unroll
  for (int j = 0; j < 16; ++j) sw[j * 33 + lane] = v[j];
  __syncwarp();
  float* y = static_cast<float*>(p.Y);
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int idx = i * 32 + lane;
    const int c = idx >> 3, k = (idx & 7) * 4;  // token c, features f0 + k .. f0 + k + 3
    if (m0 + c < p.M && f0 + k < p.N) {
      const float* s = sw + c * 33 + k;
      red_add_v4(y + static_cast<size_t>(m0 + c) * p.ldy + f0 + k, make_float4(s[0], s[1], s[2], s[3]));
    }
  }
  __syncwarp();
}

__device__ __forceinline__ bool bar_any(int id, int nthreads, bool pred) {
  uint32_t r;
  asm volatile(
      "{\n\t.reg .pred pi, po;\n\t"
      "setp.ne.u32 pi, %1, 0;\n\t"
      "bar.red.or.pred po, %2, %3, pi;\n\t"
      "selp.u32 %0, 1, 0, po;\n\t}"
      : "=r"(r)
      : "r"(static_cast<uint32_t>(pred)), "r"(id), "r"(nthreads)
      : "memory");
  return r != 0;
}


__global__ void __launch_bounds__(THREADS, CTAS_PER_SM) tc_linear_kernel(const __grid_constant__ TcLinearParams p) {
  if (p.skip) {
    // the flag is written by the previous kernel: read it after the dependency wait,
    // before any weight is requested (a skipped launch streams nothing)
    pdl_wait();
    if (*reinterpret_cast<const volatile int*>(p.skip)) {
      pdl_trigger();
      return;
    }
  }
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  const int a_atom = BM * ATOM * 2;     // one 128 x 64 weight box
  const int b_atom = p.BN * ATOM * 2;  // one BN x 64 activation box
  const int b_bytes = b_atom * BKA;
  const int stage_bytes = a_atom * BKA + (p.has_lo ? 2 : 1) * b_bytes;
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + p.stages * stage_bytes);
  uint64_t* empty = full + MAX_STAGES;
  uint64_t* tfull = empty + MAX_STAGES;
  uint64_t* tempty = tfull + 2;
  uint64_t* drain = tempty + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain + 1);
  int* s_abort = reinterpret_cast<int*>(tmem_slot + 1);
  int* s_last = s_abort + 1;
  float* s_red = reinterpret_cast<float*>(smem + p.stages * stage_bytes + 1024);  // [4 warps][16][33]

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    for (int s = 0; s < p.stages; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&tfull[b], 1);
      mbar_init(&tempty[b], 128);
    }
    mbar_init(drain, 1);
    *s_abort = 0;
    *s_last = 0;
    mbar_fence_init();
  }
  // Programmatic dependent launch: every thread calls pdl_trigger() only after its own
  // pdl_wait(), so a dependent that starts early knows that every kernel before this
  // one is complete (it may read their outputs before its own wait).
  if (warp == 0 && lane == 0) {
    prefetch_tensormap(&p.tmA);
    if (p.ft_split < p.feat_tiles) prefetch_tensormap(&p.tmA2);
    prefetch_tensormap(&p.tmB);
    if (p.has_lo) prefetch_tensormap(&p.tmB2);
  }
  if (warp == 1) tmem_alloc(tmem_slot, p.tmem_cols);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;

  const uint32_t U = static_cast<uint32_t>(p.units);
  const uint32_t G = gridDim.x;
  const int cta = blockIdx.x;
  const uint32_t u_begin = unit_begin(cta, U, G);
  const uint32_t u_end = unit_begin(cta + 1, U, G);
  const uint32_t KB = p.kblocks;
  volatile int* abort = s_abort;

  if (warp == 0) {
    if (lane == 0) {
      // ---------------- TMA producer ----------------
      const uint64_t pol_w = policy_evict_first();
      int stage = 0;
      uint32_t phase = 0;
      uint32_t issued_mask = 0, issued_par = 0;
      auto load_a = [&](uint32_t u, uint8_t* sa, uint64_t* bar) {
        const int t = static_cast<int>(u / KB), kb = static_cast<int>(u % KB);
        const int ft = t / p.tok_tiles;
        const bool second = ft >= p.ft_split;
        const CUtensorMap* map = second ? &p.tmA2 : &p.tmA;
        const int row = (second ? ft - p.ft_split : ft) * BM;
#pragma unroll
        for (int a = 0; a < BKA; ++a) tma_load_2d_hint(sa + a * a_atom, map, kb * BK + a * ATOM, row, bar, pol_w);
      };
      auto load_b = [&](uint32_t u, uint8_t* sb, uint64_t* bar) {
        const int t = static_cast<int>(u / KB), kb = static_cast<int>(u % KB);
        const int tt = t % p.tok_tiles;
#pragma unroll
        for (int a = 0; a < BKA; ++a) {
          tma_load_2d(sb + a * b_atom, &p.tmB, kb * BK + a * ATOM, tt * p.BN, bar);
          if (p.has_lo) tma_load_2d(sb + b_bytes + a * b_atom, &p.tmB2, kb * BK + a * ATOM, tt * p.BN, bar);
        }
      };
      // The weights do not depend on earlier kernels: request the first stages' weight
      // tiles before waiting for the previous kernel, then their activation tiles.  Two
      // stages, not the whole ring: the row kernel that usually runs meanwhile reads its
      // input from L2 behind these requests (measured: 1 stage 4.45, 2 stages 4.40, 3
      // stages 4.42 ms per 7B step).
      const uint32_t npre = min(static_cast<uint32_t>(min(p.stages, CHIMERA_LIN_PRE_STAGES)), u_end - u_begin);
      for (uint32_t i = 0; i < npre; ++i) {
        uint8_t* sa = smem + i * stage_bytes;
        mbar_arrive_expect_tx(&full[i], static_cast<uint32_t>(stage_bytes));
        load_a(u_begin + i, sa, &full[i]);
        issued_mask |= 1u << i;
      }
      pdl_wait();
      pdl_trigger();
      for (uint32_t i = 0; i < npre; ++i) load_b(u_begin + i, smem + i * stage_bytes + a_atom * BKA, &full[i]);
      stage = static_cast<int>(npre % p.stages);
      phase = (npre == static_cast<uint32_t>(p.stages)) ? 1u : 0u;
      for (uint32_t u = u_begin + npre; u < u_end && !*abort; ++u) {
        if (!mbar_wait(&empty[stage], phase ^ 1u, abort, p.wait_ns)) break;
        uint8_t* sa = smem + stage * stage_bytes;
        mbar_arrive_expect_tx(&full[stage], static_cast<uint32_t>(stage_bytes));
        load_a(u, sa, &full[stage]);
        load_b(u, sa + a_atom * BKA, &full[stage]);
        issued_mask |= 1u << stage;
        issued_par = (issued_par & ~(1u << stage)) | (phase << stage);
        if (++stage == p.stages) {
          stage = 0;
          phase ^= 1u;
        }
      }
      if (*abort) {
        // let copies that are still in flight land before the CTA exits
        for (int s = 0; s < p.stages; ++s)
          if (issued_mask >> s & 1u) mbar_wait_plain(&full[s], issued_par >> s & 1u, 200000000ull);
      }
    } else {
      pdl_wait();
      pdl_trigger();
    }
  } else if (warp == 1) {
    pdl_wait();
    pdl_trigger();
    if (lane == 0) {
      // ---------------- MMA issuer ----------------
      const uint32_t idesc = idesc_bf16_m128(p.BN);
      int stage = 0;
      uint32_t phase = 0;
      int buf = 0;
      uint32_t aphase = 0;
      for (uint32_t u = u_begin; u < u_end && !*abort;) {
        const int t = static_cast<int>(u / KB);
        const uint32_t seg_end = min(u_end, static_cast<uint32_t>(t + 1) * KB);
        if (!mbar_wait(&tempty[buf], aphase ^ 1u, abort, p.wait_ns)) break;
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + buf * p.acc_stride;
        bool first = true;
        for (; u < seg_end; ++u) {
          if (!mbar_wait(&full[stage], phase, abort, p.wait_ns)) break;
          tc_fence_after();
          const uint32_t sa = smem_u32(smem + stage * stage_bytes);
          const uint32_t sb = sa + a_atom * BKA;
#pragma unroll
          for (int a = 0; a < BKA; ++a) {
#pragma unroll
            for (int k = 0; k < ATOM / UK; ++k) {
              const uint64_t adesc = sw128_desc(sa + a * a_atom + k * 32);
              tc_mma_bf16(d_tmem, adesc, sw128_desc(sb + a * b_atom + k * 32), idesc,
                          (first && a == 0 && k == 0) ? 0u : 1u);
              if (p.has_lo) tc_mma_bf16(d_tmem, adesc, sw128_desc(sb + b_bytes + a * b_atom + k * 32), idesc, 1u);
            }
          }
          first = false;
          tc_commit(&empty[stage]);
          if (++stage == p.stages) {
            stage = 0;
            phase ^= 1u;
          }
        }
        tc_commit(&tfull[buf]);
        buf ^= 1;
        if (buf == 0) aphase ^= 1u;
      }
      if (*abort) {
        // every MMA issued so far must complete before TMEM is released
        tc_commit(drain);
        mbar_wait_plain(drain, 0, 200000000ull);
      }
    }
  } else {
    // ---------------- epilogue (warps 2..5, TMEM lanes 32*(warp%4) ..) ----------------
    pdl_wait();  // Y, the split workspace and the counters are shared with earlier kernels
    pdl_trigger();
    if (p.zero) {  // this CTA's share (float4s) of a later linear's accumulator
      const long long n4 = p.zero_floats / 4, per = (n4 + G - 1) / G;
      float4* z = reinterpret_cast<float4*>(p.zero);
      for (long long i = cta * per + (threadIdx.x - 64); i < min(n4, (cta + 1) * per); i += 128)
        z[i] = make_float4(0.f, 0.f, 0.f, 0.f);
    }
    const int q = warp & 3;
    const int row = q * 32 + lane;
    int buf = 0;
    uint32_t aphase = 0;
    for (uint32_t u = u_begin; u < u_end;) {
      const int t = static_cast<int>(u / KB);
      const uint32_t seg_end = min(u_end, static_cast<uint32_t>(t + 1) * KB);
      u = seg_end;
      const bool ok = mbar_wait(&tfull[buf], aphase, abort, p.wait_ns);
      if (bar_any(1, 128, !ok)) break;
      tc_fence_after();
      const int ft = t / p.tok_tiles, tt = t % p.tok_tiles;
      const uint32_t tu0 = static_cast<uint32_t>(t) * KB;
      const int c_first = cta_of_unit(tu0, U, G);
      const int c_last = cta_of_unit(tu0 + KB - 1, U, G);
      const int nparts = c_last - c_first + 1;
      const int f = ft * BM + row;
      const int m0 = tt * p.BN;
      const uint32_t tbase = tmem_base + (static_cast<uint32_t>(q * 32) << 16) + buf * p.acc_stride;
      if (nparts == 1 || p.epi == EPI_RESID) {
        for (int c0 = 0; c0 < p.BN; c0 += 16) {
          float v[16];
          tmem_ld_16(tbase + c0, v);
          if (p.vec_red)
            epi_red16(p, m0 + c0, ft * BM + q * 32, lane, v, s_red + q * 16 * 33);
          else
            epi_store16(p, m0 + c0, f, v);
        }
        tc_fence_before();
        mbar_arrive(&tempty[buf]);
      } else {
        const int my_slot = 2 * cta + ((u_begin / KB == static_cast<uint32_t>(t)) ? 0 : 1);
        float* wsp = p.ws + static_cast<size_t>(my_slot) * BM * p.BN;
        for (int c0 = 0; c0 < p.BN; c0 += 16) {
          float v[16];
          tmem_ld_16(tbase + c0, v);
#pragma unroll
          for (int j = 0; j < 16; ++j) __stcg(&wsp[(c0 + j) * BM + row], v[j]);
        }
        tc_fence_before();
        mbar_arrive(&tempty[buf]);
        __threadfence();
        named_bar(1, 128);
        if (threadIdx.x == 64) {
          const int old = atomicAdd(&p.counters[t], 1);
          *s_last = (old == nparts - 1) ? 1 : 0;
        }
        named_bar(1, 128);
        if (*s_last) {
          __threadfence();
          // slot of every contributor, computed once (contributor c2 > c_first starts
          // inside tile t, so only c_first can hold the tile in its second slot)
          const int slot_first = 2 * c_first + ((unit_begin(c_first, U, G) / KB == static_cast<uint32_t>(t)) ? 0 : 1);
          for (int c0 = 0; c0 < p.BN; c0 += 16) {
            if (m0 + c0 >= p.M) break;
            float acc[16];
#pragma unroll
            for (int j = 0; j < 16; ++j) acc[j] = 0.f;
            // partials summed in contributor order (deterministic); up to four
            // contributors' loads in flight at once
            for (int cc = c_first; cc <= c_last; cc += 4) {
              float v[4][16];
#pragma unroll
              for (int q4 = 0; q4 < 4; ++q4) {
                if (cc + q4 <= c_last) {
                  const int c2 = cc + q4;
                  const int sl = c2 == c_first ? slot_first : 2 * c2;
                  const float* src = p.ws + static_cast<size_t>(sl) * BM * p.BN + static_cast<size_t>(c0) * BM + row;
#pragma unroll
                  for (int j = 0; j < 16; ++j) v[q4][j] = __ldcg(src + j * BM);
                }
              }
#pragma unroll
              for (int q4 = 0; q4 < 4; ++q4)
                if (cc + q4 <= c_last) {
#pragma unroll
                  for (int j = 0; j < 16; ++j) acc[j] += v[q4][j];
                }
            }
            epi_store16(p, m0 + c0, f, acc);
          }
          if (threadIdx.x == 64) p.counters[t] = 0;
        }
        named_bar(1, 128);
      }
      buf ^= 1;
      if (buf == 0) aphase ^= 1u;
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_base, p.tmem_cols);
  }
  if (threadIdx.x == 0 && *abort) atomicOr(p.err, ERR_TIMEOUT);
}

// ----------------------------------------------------------------------------
// host side
// ----------------------------------------------------------------------------
typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                  const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                  const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
  static EncodeTiledFn fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* ptr = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(ptr);
  });
  return fn;
}

}  // namespace

int encode_2d_bf16(CUtensorMap* map, const void* base, uint64_t inner, uint64_t outer,
                   uint64_t pitch_elems, uint32_t box_inner, uint32_t box_outer) {
  EncodeTiledFn fn = encode_fn();
  if (!fn) return -1;
  cuuint64_t dims[2] = {inner, outer};
  cuuint64_t strides[1] = {pitch_elems * 2};
  cuuint32_t box[2] = {box_inner, box_outer};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides,
                  box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                  CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS ? 0 : -2;
}

namespace {

uint32_t pow2ceil(uint32_t v) {
  uint32_t r = 1;
  while (r < v) r <<= 1;
  return r;
}

}  // namespace

int tc_num_sms() {
  int dev = 0, n = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
  return n > 0 ? n : 1;
}

size_t tc_ws_floats(int max_bn) {
  return static_cast<size_t>(tc_num_sms()) * CTAS_PER_SM * 2 * BM * static_cast<size_t>(max_bn);
}

int tc_max_tiles() { return MAX_TILES; }


int tc_linear_plan(TcLinearPlan* plan, int M, int N, int K, const void* X, const void* X_lo, int ldx,
                   const void* W, void* Y, void* Y_lo, int ldy, int epi, int out_f32, float* ws,
                   int* counters, int* err, char* msg, size_t msg_len, const void* W2, int N2,
                   float* zero, long long zero_floats) {
  auto fail = [&](const char* m) {
    if (msg && msg_len) snprintf(msg, msg_len, "linear(M=%d,N=%d,K=%d): %s", M, N, K, m);
    return -1;
  };
  if (M < 1 || N < 1 || K < 8) return fail("empty or too-small shape");
  if (K % 8 != 0 || ldx % 8 != 0) return fail("K and the row pitch of X must be multiples of 8");
  if (ldx < K || ldy < N) return fail("row pitch smaller than the row");
  if ((reinterpret_cast<uintptr_t>(X) & 15) || (reinterpret_cast<uintptr_t>(W) & 15) ||
      (reinterpret_cast<uintptr_t>(X_lo) & 15))
    return fail("X, X_lo and W must be 16-byte aligned");
  if (epi == EPI_RESID && !out_f32) return fail("accumulating epilogue needs an fp32 output");
  if (zero && ((zero_floats & 3) || (reinterpret_cast<uintptr_t>(zero) & 15)))
    return fail("the buffer to clear must be 16-byte aligned and a multiple of 4 floats");
  if (W2 && (N % BM != 0 || N2 < 1 || (reinterpret_cast<uintptr_t>(W2) & 15)))
    return fail("second weight needs N % 128 == 0 and a 16-byte aligned W2");
  const int N1 = N;
  if (W2) N += N2;
  if (ldy < N) return fail("row pitch of Y smaller than the two outputs");
  TcLinearParams& p = plan->p;
  memset(&p, 0, sizeof(p));
  p.M = M;
  p.N = N;
  p.K = K;
  p.has_lo = X_lo ? 1 : 0;
  // token tile: all rows when the ring still holds at least two stages, else halves
  p.BN = M <= MAX_BN ? ((M + 15) / 16) * 16 : MAX_BN;
  while (p.BN > 16 && PIPE_SMEM / (BM * BK * 2 + (p.has_lo ? 2 : 1) * p.BN * BK * 2) < 2)
    p.BN = ((p.BN / 2 + 15) / 16) * 16;
  p.tok_tiles = (M + p.BN - 1) / p.BN;
  p.feat_tiles = (N + BM - 1) / BM;
  p.ft_split = W2 ? N1 / BM : p.feat_tiles;
  p.kblocks = (K + BK - 1) / BK;
  if (static_cast<long long>(p.feat_tiles) * p.tok_tiles > MAX_TILES) return fail("too many tiles");
  p.units = static_cast<long long>(p.feat_tiles) * p.tok_tiles * p.kblocks;
  if (p.units * (tc_num_sms() * CTAS_PER_SM + 1) >= (1ll << 32)) return fail("too many work units");
  p.has_lo = X_lo ? 1 : 0;
  const int stage_bytes = BM * BK * 2 + (p.has_lo ? 2 : 1) * p.BN * BK * 2;
  p.stages = PIPE_SMEM / stage_bytes;
  if (p.stages > MAX_STAGES) p.stages = MAX_STAGES;
  if (p.stages < 2) return fail("token tile too large");
  p.epi = epi;
  p.out_f32 = out_f32;
  p.Y = Y;
  p.Y2 = out_f32 ? nullptr : Y_lo;
  p.ldy = ldy;
  p.zero = zero;
  p.zero_floats = zero ? zero_floats : 0;
  p.ws = ws;
  p.counters = counters;
  p.err = err;
  p.wait_ns = g_lin_wait_ns.load();
  p.acc_stride = pow2ceil(static_cast<uint32_t>(p.BN));
  p.tmem_cols = pow2ceil(2 * p.acc_stride);
  if (p.tmem_cols < 32) p.tmem_cols = 32;
  if (p.tmem_cols > 512) return fail("accumulators exceed tensor memory");
  if (encode_2d_bf16(&p.tmA, W, K, N1, K, ATOM, BM) != 0) return fail("tensor map of W");
  if (W2 && encode_2d_bf16(&p.tmA2, W2, K, N2, K, ATOM, BM) != 0) return fail("tensor map of W2");
  if (encode_2d_bf16(&p.tmB, X, K, M, ldx, ATOM, p.BN) != 0) return fail("tensor map of X");
  if (X_lo && encode_2d_bf16(&p.tmB2, X_lo, K, M, ldx, ATOM, p.BN) != 0) return fail("tensor map of X_lo");
  const int sms = tc_num_sms() * CTAS_PER_SM;
  plan->grid = static_cast<int>(p.units < sms ? p.units : sms);
  // float4 reductions need 16-byte aligned rows of Y and whole float4 runs of features
  p.vec_red = (epi == EPI_RESID && (reinterpret_cast<uintptr_t>(Y) & 15) == 0 && ldy % 4 == 0 && N % 4 == 0) ? 1 : 0;
  plan->smem = 1024 + static_cast<size_t>(p.stages) * stage_bytes + 1024 + 4 * 16 * 33 * sizeof(float);
  plan->weight_bytes = 2.0 * N * K;
  return 0;
}

namespace {
// The kernel's dynamic shared memory limit is an attribute of the device that is
// current when it is set: raise it once per device, before the first launch there.
constexpr int LIN_MAX_DEVICES = 64;
std::mutex g_attr_mu;
bool g_attr_set[LIN_MAX_DEVICES];
}  // namespace

std::atomic<unsigned long long> g_lin_wait_ns{kDefaultWaitNs};

cudaError_t tc_linear_launch(const TcLinearPlan& plan, cudaStream_t s) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= LIN_MAX_DEVICES) return cudaErrorInvalidDevice;
  {
    std::lock_guard<std::mutex> lk(g_attr_mu);
    if (!g_attr_set[dev]) {
      e = cudaFuncSetAttribute(tc_linear_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, 227 * 1024);
      if (e != cudaSuccess) return e;
      g_attr_set[dev] = true;
    }
  }
  launch_pdl(tc_linear_kernel, dim3(plan.grid), dim3(THREADS), plan.smem, s, plan.p);
  return cudaGetLastError();
}

}  // namespace chimera
