// Persistent chain of a decoder block's weight-streaming linears and the row
// operations between them, in one launch (sm_103a, tcgen05 + TMA).
//
// A chain is a short program of steps, e.g. for the tree verify of one layer boundary:
//
//   O projection (+ residual) | RMSNorm | gate|up | SwiGLU | down (+ residual) |
//   RMSNorm of the next layer | its QKV projection
//
// Every CTA (one per SM, all resident: grid = SM count) takes a stream-K share of
// every linear's (feature tile, token tile, K block) units, and a share of the rows
// of every row step.  Steps that consume another step's output wait for it through a
// grid-wide arrival counter (one per step, bounded waits); nothing else is ordered.
// The weights do not depend on anything, so the TMA producer of each CTA keeps
// requesting the weight tiles of its next units across step boundaries: while the
// CTAs wait for a norm or for the last partial sums of a linear, HBM keeps streaming
// into the shared-memory ring (the activation half of a stage is requested only once
// its producing step has completed).
//
// Roles (192 threads): warp 0 lane 0 issues TMA loads, warp 1 lane 0 issues
// tcgen05.mma into one of two tensor-memory accumulators, warps 2..5 drain the other
// accumulator into fp32 outputs with vector red.global.add and run the row steps.
//
// Ordering: a step's contributions are published by every epilogue thread's
// __threadfence, a named barrier and one atomicAdd on the step's counter; consumers
// read the counter with ld.acquire.gpu (the producer then fences the async proxy
// before its TMA reads) and read other CTAs' data with L1-bypassing loads.  The CTA
// that arrives last on the launch's final counter resets all counters to zero for the
// next launch.  The launch lets its dependents start only after its own dependency
// wait, so a dependent that reads before its own wait sees every earlier kernel done.
//
// Measured on a GB300 (7B shape, 64 tree rows): a layer-boundary chain takes ~141 us for
// 405 MB (2.9 TB/s), against ~100 us for the same linears and row kernels launched
// separately.  Every step waits for the slowest CTA of the previous one (a 3-6 us
// spread at each boundary), and a row step under full HBM load costs 6-9 us including
// its two grid-wide counter rounds; separate launches hide those tails because the next
// kernel starts on whichever SMs free up first.  The chain is therefore an option
// (config field fused_chain), not the default.
#include <cstdio>
#include <cstring>
#include <mutex>

#include "common.cuh"
#include "launch.cuh"
#include "kernels.h"

namespace chimera {
namespace {

constexpr int BM = 128;             // weight rows per tile (UMMA M)
constexpr int ATOM = 64;            // bf16 per 128-byte swizzle atom
constexpr int BKA = 2;              // atoms per stage
constexpr int BK = ATOM * BKA;      // K per stage
constexpr int UK = 16;              // UMMA K (16-bit inputs)
constexpr int MAX_STAGES = 12;
constexpr int THREADS = 192;
constexpr int PIPE_SMEM = 200 * 1024;
constexpr int NORM_VEC = 16;        // float4 per epilogue thread: d <= 8192

__device__ __forceinline__ uint32_t unit_begin(uint32_t c, uint32_t U, uint32_t G) {
  return static_cast<uint32_t>((static_cast<unsigned long long>(c) * U) / G);
}

__device__ __forceinline__ int ld_acquire(const int* p) {
  int v;
  asm volatile("ld.acquire.gpu.global.b32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}

__device__ __forceinline__ void fence_proxy_async_global() {
  asm volatile("fence.proxy.async.global;" ::: "memory");
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

// fp32 outputs of 32 feature rows (f0 ..) x 16 token columns (m0 ..) added into Y with
// float4 reductions (a shared-memory transpose gives each lane four consecutive features)
__device__ __forceinline__ void red16(const ChainGemm& g, int M, int m0, int f0, int lane, const float (&v)[16],
                                      float* sw) {
#pragma unroll
  for (int j = 0; j < 16; ++j) sw[j * 33 + lane] = v[j];
  __syncwarp();
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int idx = i * 32 + lane;
    const int c = idx >> 3, k = (idx & 7) * 4;
    if (m0 + c < M && f0 + k < g.N) {
      const float* s = sw + c * 33 + k;
      red_add_v4(g.Y + static_cast<size_t>(m0 + c) * g.ldy + f0 + k,
                make_float4(s[0], s[1], s[2], s[3]));
    }
  }
  __syncwarp();
}

__device__ __forceinline__ float4 ldcg4(const float* p) { return __ldcg(reinterpret_cast<const float4*>(p)); }

__device__ __forceinline__ float4 gain4(const bf16* g, int i) {
  const uint2 u = *reinterpret_cast<const uint2*>(g + i);
  const bf16* h = reinterpret_cast<const bf16*>(&u);
  return make_float4(__bfloat162float(h[0]), __bfloat162float(h[1]), __bfloat162float(h[2]), __bfloat162float(h[3]));
}

__device__ __forceinline__ void store_split4(bf16* hi, bf16* lo, size_t i, float4 v) { store_act4(hi, lo, i, v); }

__global__ void __launch_bounds__(THREADS, 1) chain_kernel(const __grid_constant__ ChainParams p) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  const int a_atom = BM * ATOM * 2;
  const int b_atom = p.BN * ATOM * 2;
  const int b_bytes = b_atom * BKA;
  const int stage_bytes = a_atom * BKA + (p.has_lo ? 2 : 1) * b_bytes;
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + p.stages * stage_bytes);
  uint64_t* empty = full + MAX_STAGES;
  uint64_t* tfull = empty + MAX_STAGES;
  uint64_t* tempty = tfull + 2;
  uint64_t* drain = tempty + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain + 1);
  int* s_abort = reinterpret_cast<int*>(tmem_slot + 1);
  float* s_sum = reinterpret_cast<float*>(s_abort + 4);                            // [4] norm partials
  float* s_red = reinterpret_cast<float*>(smem + p.stages * stage_bytes + 1024);  // [4][16][33]

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
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
    mbar_fence_init();
  }
  if (warp == 0 && lane == 0) {
    for (int g = 0; g < p.n_gemm; ++g) {
      prefetch_tensormap(&p.gemm[g].tmA);
      if (p.gemm[g].ft_split < p.gemm[g].feat_tiles) prefetch_tensormap(&p.gemm[g].tmA2);
      prefetch_tensormap(&p.gemm[g].tmB);
      if (p.has_lo) prefetch_tensormap(&p.gemm[g].tmB2);
    }
  }
  if (warp == 1) tmem_alloc(tmem_slot, p.tmem_cols);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  const uint32_t G = gridDim.x;
  const uint32_t cta = blockIdx.x;
  volatile int* abort = s_abort;

  // this CTA's unit range of every linear
  uint32_t ub[CHAIN_MAX_GEMM], ue[CHAIN_MAX_GEMM];
#pragma unroll
  for (int g = 0; g < CHAIN_MAX_GEMM; ++g) {
    ub[g] = g < p.n_gemm ? unit_begin(cta, p.gemm[g].units, G) : 0u;
    ue[g] = g < p.n_gemm ? unit_begin(cta + 1, p.gemm[g].units, G) : 0u;
  }

  if (warp == 0) {
    if (lane == 0) {
      // ---------------- TMA producer ----------------
      const uint64_t pol_w = policy_evict_first();
      uint32_t total = 0;
      for (int g = 0; g < p.n_gemm; ++g) total += ue[g] - ub[g];
      // cursors over the CTA's units of all linears, in step order
      int wg = 0, xg = 0;
      uint32_t wu = ub[0], xu = ub[0];
      uint32_t wq = 0, xq = 0;
      int xg_ready = -1;  // linear whose activation dependency is known complete
      auto norm_cursor = [&](int& g, uint32_t& u) {
        while (g < p.n_gemm && u >= ue[g]) {
          ++g;
          if (g < p.n_gemm) u = ub[g];
        }
      };
      norm_cursor(wg, wu);
      norm_cursor(xg, xu);
      auto issue_w = [&](uint32_t q, int g, uint32_t u) {
        const ChainGemm& gm = p.gemm[g];
        const int s = static_cast<int>(q % p.stages);
        uint8_t* sa = smem + s * stage_bytes;
        mbar_arrive_expect_tx(&full[s], static_cast<uint32_t>(stage_bytes));
        const uint32_t KB = gm.kblocks;
        const int t = static_cast<int>(u / KB), kb = static_cast<int>(u % KB);
        const int ft = t / p.tok_tiles;
        const bool second = ft >= gm.ft_split;
        const CUtensorMap* map = second ? &gm.tmA2 : &gm.tmA;
        const int row = (second ? ft - gm.ft_split : ft) * BM;
#pragma unroll
        for (int a = 0; a < BKA; ++a) tma_load_2d_hint(sa + a * a_atom, map, kb * BK + a * ATOM, row, &full[s], pol_w);
      };
      auto issue_x = [&](uint32_t q, int g, uint32_t u) {
        const ChainGemm& gm = p.gemm[g];
        const int s = static_cast<int>(q % p.stages);
        uint8_t* sb = smem + s * stage_bytes + a_atom * BKA;
        const uint32_t KB = gm.kblocks;
        const int t = static_cast<int>(u / KB), kb = static_cast<int>(u % KB);
        const int tt = t % p.tok_tiles;
#pragma unroll
        for (int a = 0; a < BKA; ++a) {
          tma_load_2d(sb + a * b_atom, &gm.tmB, kb * BK + a * ATOM, tt * p.BN, &full[s]);
          if (p.has_lo) tma_load_2d(sb + b_bytes + a * b_atom, &gm.tmB2, kb * BK + a * ATOM, tt * p.BN, &full[s]);
        }
      };
      // weight tiles of the first stages before the dependency wait
      while (wq < total && wq < static_cast<uint32_t>(p.stages)) {
        issue_w(wq, wg, wu);
        ++wq;
        ++wu;
        norm_cursor(wg, wu);
      }
      pdl_wait();
      pdl_trigger();
      uint64_t t_last = global_timer_ns();
      while (xq < total && !*abort) {
        bool moved = false;
        // activation tile of unit xq once its producing step has completed
        if (xq < wq) {
          bool ready = xg_ready == xg;
          if (!ready) {
            const int st = p.gemm_step[xg];
            const int w = p.wait[st];
            ready = w < 0 || ld_acquire(p.bars + w) >= static_cast<int>(G);
            if (ready) {
              fence_proxy_async_global();
              xg_ready = xg;
            }
          }
          if (ready) {
            issue_x(xq, xg, xu);
            ++xq;
            ++xu;
            norm_cursor(xg, xu);
            moved = true;
          }
        }
        // weight tile of unit wq once its ring slot is free (unit wq - stages consumed)
        if (wq < total && wq < xq + static_cast<uint32_t>(p.stages)) {
          const int s = static_cast<int>(wq % p.stages);
          if (mbar_test(&empty[s], ((wq / p.stages) - 1u) & 1u)) {
            issue_w(wq, wg, wu);
            ++wq;
            ++wu;
            norm_cursor(wg, wu);
            moved = true;
          }
        }
        if (moved) {
          t_last = global_timer_ns();
        } else if (global_timer_ns() - t_last > p.wait_ns) {
          *abort = 1;
        }
      }
      if (*abort) {
        // every started stage must land before the CTA exits: request the activation
        // half of the units whose weights are in flight too (in-bounds reads of
        // whatever the buffer holds), then wait for the last `stages` units
        while (xq < wq) {
          issue_x(xq, xg, xu);
          ++xq;
          ++xu;
          norm_cursor(xg, xu);
        }
        for (uint32_t q = (wq > static_cast<uint32_t>(p.stages) ? wq - p.stages : 0u); q < wq; ++q)
          mbar_wait_plain(&full[q % p.stages], (q / p.stages) & 1u, 200000000ull);
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
      uint32_t q = 0;
      int buf = 0;
      uint32_t aphase = 0;
      for (int g = 0; g < p.n_gemm && !*abort; ++g) {
        const uint32_t KB = p.gemm[g].kblocks;
        for (uint32_t u = ub[g]; u < ue[g] && !*abort;) {
          const uint32_t t = u / KB;
          const uint32_t seg_end = min(ue[g], (t + 1) * KB);
          if (!mbar_wait(&tempty[buf], aphase ^ 1u, abort, p.wait_ns)) break;
          tc_fence_after();
          const uint32_t d_tmem = tmem_base + buf * p.acc_stride;
          bool first = true;
          for (; u < seg_end; ++u, ++q) {
            const int s = static_cast<int>(q % p.stages);
            if (!mbar_wait(&full[s], (q / p.stages) & 1u, abort, p.wait_ns)) break;
            tc_fence_after();
            const uint32_t sa = smem_u32(smem + s * stage_bytes);
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
            tc_commit(&empty[s]);
          }
          tc_commit(&tfull[buf]);
          buf ^= 1;
          if (buf == 0) aphase ^= 1u;
        }
      }
      if (*abort) {
        tc_commit(drain);
        mbar_wait_plain(drain, 0, 200000000ull);
      }
    }
  } else {
    // ---------------- epilogue and row steps (warps 2..5, 128 threads) ----------------
    pdl_wait();
    pdl_trigger();
    const int et = threadIdx.x - 64;  // 0..127
    const int qd = warp & 3;          // TMEM sub-partition of this warp
    int buf = 0;
    uint32_t aphase = 0;
    bool dead = false;
    // wait until step `w` has all G arrivals (one thread polls, bounded)
    auto wait_step = [&](int w) -> bool {
      int ok = 1;
      if (w >= 0 && et == 0) {
        const uint64_t t0 = global_timer_ns();
        while (ld_acquire(p.bars + w) < static_cast<int>(G)) {
          if (*abort || global_timer_ns() - t0 > p.wait_ns) {
            *abort = 1;
            ok = 0;
            break;
          }
        }
      }
      const bool bad = bar_any(1, 128, !ok);
      __threadfence();
      return !bad;
    };
    auto signal = [&](int s) {
      __threadfence();
      named_bar(1, 128);
      if (et == 0) atomicAdd(p.bars + s, 1);
    };
    for (int s = 0; s < p.n_steps && !dead; ++s) {
      const int kind = p.kind[s];
      if (kind == CH_GEMM) {
        const int g = p.idx[s];
        const ChainGemm& gm = p.gemm[g];
        const uint32_t KB = gm.kblocks;
        for (uint32_t u = ub[g]; u < ue[g];) {
          const uint32_t t = u / KB;
          u = min(ue[g], (t + 1) * KB);
          const bool ok = mbar_wait(&tfull[buf], aphase, abort, p.wait_ns);
          if (bar_any(1, 128, !ok)) {
            dead = true;
            break;
          }
          tc_fence_after();
          const int ft = static_cast<int>(t) / p.tok_tiles, tt = static_cast<int>(t) % p.tok_tiles;
          const uint32_t tbase = tmem_base + (static_cast<uint32_t>(qd * 32) << 16) + buf * p.acc_stride;
          for (int c0 = 0; c0 < p.BN; c0 += 16) {
            float v[16];
            tmem_ld_16(tbase + c0, v);
            red16(gm, p.M, tt * p.BN + c0, ft * BM + qd * 32, lane, v, s_red + qd * 16 * 33);
          }
          tc_fence_before();
          mbar_arrive(&tempty[buf]);
          buf ^= 1;
          if (buf == 0) aphase ^= 1u;
        }
        if (dead) break;
        signal(s);
        continue;
      }
      if (!wait_step(p.wait[s])) {
        dead = true;
        break;
      }
      const ChainRow& r = p.row[p.idx[s]];
      if (kind == CH_NORM) {
        // RMSNorm of rows cta, cta + G, ...: y = x / sqrt(mean(x^2) + eps) * g, written as
        // the bf16 hi + lo operand (and an fp32 copy); row r of Z is cleared
        for (int row = static_cast<int>(cta); row < r.rows; row += static_cast<int>(G)) {
          const float* x = r.X + static_cast<size_t>(row) * r.ldx;
          float4 v[NORM_VEC];
          float ss = 0.f;
#pragma unroll
          for (int k = 0; k < NORM_VEC; ++k) {
            const int i = (et + k * 128) * 4;
            v[k] = i < r.cols ? ldcg4(x + i) : make_float4(0.f, 0.f, 0.f, 0.f);
            ss += v[k].x * v[k].x + v[k].y * v[k].y + v[k].z * v[k].z + v[k].w * v[k].w;
          }
#pragma unroll
          for (int o = 16; o > 0; o >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
          if (lane == 0) s_sum[qd] = ss;
          named_bar(1, 128);
          const float tot = (s_sum[0] + s_sum[1]) + (s_sum[2] + s_sum[3]);
          named_bar(1, 128);
          const float rs = rsqrtf(tot / static_cast<float>(r.cols) + r.eps);
          const bf16* gn = static_cast<const bf16*>(r.g);
#pragma unroll
          for (int k = 0; k < NORM_VEC; ++k) {
            const int i = (et + k * 128) * 4;
            if (i < r.cols) {
              const float4 gg = gain4(gn, i);
              const float4 y = make_float4(v[k].x * rs * gg.x, v[k].y * rs * gg.y, v[k].z * rs * gg.z, v[k].w * rs * gg.w);
              store_split4(static_cast<bf16*>(r.Y), static_cast<bf16*>(r.Y_lo), static_cast<size_t>(row) * r.ldy + i, y);
              if (r.Y32) *reinterpret_cast<float4*>(r.Y32 + static_cast<size_t>(row) * r.ld32 + i) = y;
            }
          }
          if (r.Z) {
            float4* z = reinterpret_cast<float4*>(r.Z + static_cast<size_t>(row) * r.ldz);
            for (int i = et; i < r.zcols / 4; i += 128) z[i] = make_float4(0.f, 0.f, 0.f, 0.f);
          }
        }
      } else if (kind == CH_SWIGLU) {
        // h = SiLU(gate) * up over this CTA's share of the rows x F/4 float4 chunks
        const long long F4 = r.cols / 4, C = static_cast<long long>(r.rows) * F4;
        const long long c0 = static_cast<long long>(cta) * C / G, c1 = static_cast<long long>(cta + 1) * C / G;
        for (long long i = c0 + et; i < c1; i += 128) {
          const int row = static_cast<int>(i / F4), f = static_cast<int>(i % F4) * 4;
          const float* gu = r.X + static_cast<size_t>(row) * r.ldx;
          const float4 a = ldcg4(gu + f), u = ldcg4(gu + r.cols + f);
          store_split4(static_cast<bf16*>(r.Y), static_cast<bf16*>(r.Y_lo), static_cast<size_t>(row) * r.ldy + f,
                       make_float4(silu_f(a.x) * u.x, silu_f(a.y) * u.y, silu_f(a.z) * u.z, silu_f(a.w) * u.w));
        }
      } else {  // CH_COPY: rows of X into the bf16 operand Y (+ lo) and the fp32 copy Y32; Z rows cleared
        for (int row = static_cast<int>(cta); row < r.rows; row += static_cast<int>(G)) {
          const float* x = r.X + static_cast<size_t>(row) * r.ldx;
          for (int i = et * 4; i < r.cols; i += 512) {
            const float4 v = ldcg4(x + i);
            store_split4(static_cast<bf16*>(r.Y), static_cast<bf16*>(r.Y_lo), static_cast<size_t>(row) * r.ldy + i, v);
            if (r.Y32) *reinterpret_cast<float4*>(r.Y32 + static_cast<size_t>(row) * r.ld32 + i) = v;
          }
          if (r.Z) {
            float4* z = reinterpret_cast<float4*>(r.Z + static_cast<size_t>(row) * r.ldz);
            for (int i = et; i < r.zcols / 4; i += 128) z[i] = make_float4(0.f, 0.f, 0.f, 0.f);
          }
        }
      }
      signal(s);
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_base, p.tmem_cols);
  }
  if (threadIdx.x == 0) {
    if (*abort) atomicOr(p.err, ERR_TIMEOUT);
    // the last CTA to finish clears every counter of the launch (all CTAs are past
    // all their waits by now)
    __threadfence();
    const int done = atomicAdd(p.bars + CHAIN_MAX_STEPS, 1);
    if (done == static_cast<int>(G) - 1) {
      for (int i = 0; i <= CHAIN_MAX_STEPS; ++i) atomicExch(p.bars + i, 0);
      __threadfence();
    }
  }
}

// dynamic shared memory of a plan (1 KB alignment slack, stages, barriers, transpose)
size_t chain_smem(int stages, int stage_bytes) {
  return 1024 + static_cast<size_t>(stages) * stage_bytes + 1024 + 4 * 16 * 33 * sizeof(float);
}

constexpr int CH_MAX_DEVICES = 64;
std::mutex g_chain_attr_mu;
bool g_chain_attr[CH_MAX_DEVICES];

}  // namespace

int chain_plan(ChainPlan* plan, int M, int has_lo, char* msg, size_t msg_len) {
  auto fail = [&](const char* m) {
    if (msg && msg_len) snprintf(msg, msg_len, "chain(M=%d): %s", M, m);
    return -1;
  };
  memset(plan, 0, sizeof(*plan));
  ChainParams& p = plan->p;
  if (M < 1) return fail("no rows");
  p.M = M;
  p.has_lo = has_lo ? 1 : 0;
  p.BN = M <= 256 ? ((M + 15) / 16) * 16 : 256;
  while (p.BN > 16 && PIPE_SMEM / (BM * BK * 2 + (p.has_lo ? 2 : 1) * p.BN * BK * 2) < 2)
    p.BN = ((p.BN / 2 + 15) / 16) * 16;
  p.tok_tiles = (M + p.BN - 1) / p.BN;
  const int stage_bytes = BM * BK * 2 + (p.has_lo ? 2 : 1) * p.BN * BK * 2;
  p.stages = PIPE_SMEM / stage_bytes;
  if (p.stages > MAX_STAGES) p.stages = MAX_STAGES;
  if (p.stages < 2) return fail("token tile too large");
  uint32_t acc = 1;
  while (acc < static_cast<uint32_t>(p.BN)) acc <<= 1;
  p.acc_stride = acc;
  p.tmem_cols = acc * 2 < 32 ? 32 : acc * 2;
  if (p.tmem_cols > 512) return fail("accumulators exceed tensor memory");
  p.wait_ns = kDefaultWaitNs;
  plan->grid = tc_num_sms();
  plan->smem = chain_smem(p.stages, stage_bytes);
  for (int s = 0; s < CHAIN_MAX_STEPS; ++s) p.wait[s] = -1;
  return 0;
}

int chain_add_gemm(ChainPlan* plan, int wait, const void* X, const void* X_lo, int ldx, int K, const void* W,
                   int N, const void* W2, int N2, float* Y, int ldy, char* msg, size_t msg_len) {
  ChainParams& p = plan->p;
  auto fail = [&](const char* m) {
    if (msg && msg_len) snprintf(msg, msg_len, "chain linear (N=%d, K=%d): %s", N + N2, K, m);
    return -1;
  };
  if (p.n_gemm >= CHAIN_MAX_GEMM || p.n_steps >= CHAIN_MAX_STEPS) return fail("too many steps");
  if (K < 8 || K % 8 || ldx % 8 || ldx < K || N < 1) return fail("bad shape (K, ldx multiples of 8)");
  if (static_cast<bool>(X_lo) != static_cast<bool>(p.has_lo)) return fail("lo operand must match the plan");
  if ((reinterpret_cast<uintptr_t>(X) | reinterpret_cast<uintptr_t>(X_lo) | reinterpret_cast<uintptr_t>(W) |
       reinterpret_cast<uintptr_t>(W2)) & 15)
    return fail("operands must be 16-byte aligned");
  if (W2 && N % BM) return fail("a second weight needs N % 128 == 0");
  if ((reinterpret_cast<uintptr_t>(Y) & 15) || ldy % 4 || (N + N2) % 4 || ldy < N + N2)
    return fail("fp32 output rows must be 16-byte aligned runs of whole float4");
  ChainGemm& g = p.gemm[p.n_gemm];
  g.N = N + (W2 ? N2 : 0);
  g.K = K;
  g.feat_tiles = (g.N + BM - 1) / BM;
  g.ft_split = W2 ? N / BM : g.feat_tiles;
  g.kblocks = (K + BK - 1) / BK;
  const unsigned long long units = static_cast<unsigned long long>(g.feat_tiles) * p.tok_tiles * g.kblocks;
  if (units * (static_cast<unsigned long long>(plan->grid) + 1) >= (1ull << 32)) return fail("too many units");
  g.units = static_cast<uint32_t>(units);
  g.Y = Y;
  g.ldy = ldy;
  if (encode_2d_bf16(&g.tmA, W, K, N, K, ATOM, BM) != 0) return fail("tensor map of W");
  if (W2 && encode_2d_bf16(&g.tmA2, W2, K, N2, K, ATOM, BM) != 0) return fail("tensor map of W2");
  if (encode_2d_bf16(&g.tmB, X, K, p.M, ldx, ATOM, p.BN) != 0) return fail("tensor map of X");
  if (X_lo && encode_2d_bf16(&g.tmB2, X_lo, K, p.M, ldx, ATOM, p.BN) != 0) return fail("tensor map of X_lo");
  const int s = p.n_steps++;
  p.kind[s] = CH_GEMM;
  p.idx[s] = p.n_gemm;
  p.wait[s] = wait;
  p.gemm_step[p.n_gemm] = s;
  p.n_gemm++;
  plan->weight_bytes += 2.0 * (static_cast<double>(N) + (W2 ? N2 : 0)) * K;
  return s;
}

int chain_add_row(ChainPlan* plan, int kind, int wait, const ChainRow& row, char* msg, size_t msg_len) {
  ChainParams& p = plan->p;
  auto fail = [&](const char* m) {
    if (msg && msg_len) snprintf(msg, msg_len, "chain row step: %s", m);
    return -1;
  };
  if (p.n_steps >= CHAIN_MAX_STEPS || p.n_row >= CHAIN_MAX_ROW) return fail("too many steps");
  if (kind != CH_NORM && kind != CH_SWIGLU && kind != CH_COPY) return fail("unknown kind");
  if (row.cols % 4 || row.ldx % 4 || row.ldy % 4 || (row.Y32 && row.ld32 % 4) || (row.Z && (row.ldz % 4 || row.zcols % 4)))
    return fail("rows must be whole float4 runs");
  if (kind == CH_NORM && row.cols > NORM_VEC * 128 * 4) return fail("row too long for the norm");
  const int s = p.n_steps++;
  p.kind[s] = kind;
  p.idx[s] = p.n_row;
  p.wait[s] = wait;
  p.row[p.n_row++] = row;
  return s;
}

cudaError_t chain_launch(const ChainPlan& plan, cudaStream_t s) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= CH_MAX_DEVICES) return cudaErrorInvalidDevice;
  {
    std::lock_guard<std::mutex> lk(g_chain_attr_mu);
    if (!g_chain_attr[dev]) {
      e = cudaFuncSetAttribute(chain_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, 227 * 1024);
      if (e != cudaSuccess) return e;
      g_chain_attr[dev] = true;
    }
  }
  launch_pdl(chain_kernel, dim3(plan.grid), dim3(THREADS), plan.smem, s, plan.p);
  return cudaGetLastError();
}

}  // namespace chimera
