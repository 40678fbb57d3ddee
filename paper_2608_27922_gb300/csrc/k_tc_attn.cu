// Bank-reading attention on the tensor cores (bf16, d = 128):
//   O = softmax(Q [K_bank ; K_win]^T / sqrt(d)) [V_bank ; V_win]        (Sec. 3.2, Fig. 2)
// over the m_h retained bank states followed by the W window states, no mask.
//
// One CTA owns 128 queries of one head and streams 128-key tiles (bank tiles first,
// then window tiles).  Per tile:
//   S = Q K^T           tcgen05.mma into one of two 128-column TMEM buffers
//   P = exp2(S log2(e)/sqrt(d) - m)   softmax warps (thread = query row), bf16 into smem
//   O += P V            tcgen05.mma, V read as an MN-major operand, O in TMEM
// The running maximum m is raised only when a tile's maximum exceeds it by more than
// 8 (log2 units); O and the running sum are then rescaled in TMEM.  Exponentials stay
// below 2^8, and the final O / l is exact softmax algebra (the common factor cancels).
//
// Warps: 0 TMA producer, 1 MMA issuer, 2-5 softmax + output.  TMEM: S0, S1, O.
#include "dkv_internal.h"
#include "tc_ptx.cuh"

#include <climits>

namespace dkv {

bool make_map_rows(CUtensorMap* m, const void* base, int64_t rows, int64_t heads, int box_rows);

namespace {

using namespace tc;

constexpr int BQ = 128;                 // queries per CTA
constexpr int BK = 128;                 // keys per tile
constexpr int TB = 128 * 128 * 2;       // bytes of a 128 x 128 bf16 tile
constexpr int HB = TB / 2;              // one 64-column swizzle panel
constexpr int THREADS = 192;
constexpr uint32_t TMEM_COLS = 512;     // S0 [0,128), S1 [128,256), O [256,384)
constexpr uint32_t O_COL = 256;
// Q, K[2], V[2], P[2] tiles + barriers
constexpr size_t SMEM_BYTES = 1024 + TB * 7 + 256;
constexpr float RESCALE_LOG2 = 8.0f;

__device__ __forceinline__ float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

__device__ __forceinline__ uint32_t pack_bf16(float a, float b) {
  __nv_bfloat162 v = __floats2bfloat162_rn(a, b);
  return *reinterpret_cast<uint32_t*>(&v);
}

struct AttnJob {
  Bank b;
  DevLayer* L;   // sticky error word
  int Nq;
  int W;
  __nv_bfloat16* O;
  float sl2;   // log2(e) / sqrt(d)
};

__global__ void __launch_bounds__(THREADS, 1)
    tc_attend(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmKb,
              const __grid_constant__ CUtensorMap tmVb, const __grid_constant__ CUtensorMap tmKw,
              const __grid_constant__ CUtensorMap tmVw, AttnJob j) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);
  uint8_t* sQ = smem;
  uint8_t* sK = smem + TB;        // [2]
  uint8_t* sV = smem + 3 * TB;    // [2]
  uint8_t* sP = smem + 5 * TB;    // [2]
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + 7 * TB);
  uint64_t* q_full = bars + 0;
  uint64_t* k_full = bars + 1;    // [2]
  uint64_t* k_empty = bars + 3;   // [2]
  uint64_t* v_full = bars + 5;    // [2]
  uint64_t* v_empty = bars + 7;   // [2]
  uint64_t* s_full = bars + 9;    // [2]
  uint64_t* s_free = bars + 11;   // [2]
  uint64_t* p_full = bars + 13;   // [2]
  uint64_t* p_free = bars + 15;   // [2]
  uint64_t* pv_done = bars + 17;
  uint32_t* tmem_holder = reinterpret_cast<uint32_t*>(bars + 18);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_holder + 1);

  const int h = blockIdx.y;
  const int q0 = blockIdx.x * BQ;
  const int m = min(max(j.b.occ[h], 0), j.b.M_max);
  const int W = j.W;
  const int nb = (m + BK - 1) / BK;            // bank tiles
  const int nt = nb + (W + BK - 1) / BK;       // all key tiles
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    mbar_init(q_full, 1);
    for (int i = 0; i < 2; ++i) {
      mbar_init(k_full + i, 1); mbar_init(k_empty + i, 1);
      mbar_init(v_full + i, 1); mbar_init(v_empty + i, 1);
      mbar_init(s_full + i, 1); mbar_init(s_free + i, 4);
      mbar_init(p_full + i, 4); mbar_init(p_free + i, 1);
    }
    mbar_init(pv_done, 1);
    *abort_flag = 0;
    fence_barrier_init();
  }
  if (warp == 1) tmem_alloc(tmem_holder, TMEM_COLS);
  fence_before_sync();
  __syncthreads();
  fence_after_sync();
  const uint32_t tmem = *tmem_holder;

  if (warp == 0) {
    if (lane == 0 && nt > 0) {
      // ---------------- TMA producer
      prefetch_map(&tmQ);
      mbar_arrive_expect_tx(q_full, TB);
      tma_load_3d(sQ, &tmQ, q_full, 0, q0, h);
      tma_load_3d(sQ + HB, &tmQ, q_full, 64, q0, h);
      int kiss = 0, viss = 0;
      bool ok = true;
      for (int t = 0; t < nt && ok; ++t) {
        const int s = t & 1;
        const uint32_t ph = ((t >> 1) & 1) ^ 1;
        const bool bank = t < nb;
        const CUtensorMap* mk = bank ? &tmKb : &tmKw;
        const CUtensorMap* mv = bank ? &tmVb : &tmVw;
        const int row = bank ? t * BK : (t - nb) * BK;
        if (!(ok = mbar_wait(k_empty + s, ph, abort_flag))) break;
        mbar_arrive_expect_tx(k_full + s, TB);
        tma_load_3d(sK + s * TB, mk, k_full + s, 0, row, h);
        tma_load_3d(sK + s * TB + HB, mk, k_full + s, 64, row, h);
        kiss = t + 1;
        if (!(ok = mbar_wait(v_empty + s, ph, abort_flag))) break;
        mbar_arrive_expect_tx(v_full + s, TB);
        tma_load_3d(sV + s * TB, mv, v_full + s, 0, row, h);
        tma_load_3d(sV + s * TB + HB, mv, v_full + s, 64, row, h);
        viss = t + 1;
      }
      if (!ok) {
        *abort_flag = 1;
        dev_fail(j.L, DEV_TIMEOUT, 400);
      }
      volatile int no_abort = 0;
      mbar_wait(q_full, 0, &no_abort);
      for (int t = kiss > 2 ? kiss - 2 : 0; t < kiss; ++t) mbar_wait(k_full + (t & 1), (t >> 1) & 1, &no_abort);
      for (int t = viss > 2 ? viss - 2 : 0; t < viss; ++t) mbar_wait(v_full + (t & 1), (t >> 1) & 1, &no_abort);
    }
  } else if (warp == 1) {
    if (lane == 0 && nt > 0) {
      // ---------------- MMA issuer: S_t, then PV_{t-1}
      constexpr uint32_t id_s = idesc_bf16(BQ, BK);
      constexpr uint32_t id_o = idesc_bf16(BQ, 128, /*b_mn_major=*/true);
      bool ok = mbar_wait(q_full, 0, abort_flag);
      const uint32_t q_base = smem_u32(sQ);
      int pv_issued = 0;
      for (int t = 0; ok && t <= nt; ++t) {
        if (t < nt) {
          const int s = t & 1;
          if (!(ok = mbar_wait(k_full + s, (t >> 1) & 1, abort_flag))) break;
          if (!(ok = mbar_wait(s_free + s, ((t >> 1) & 1) ^ 1, abort_flag))) break;
          fence_after_sync();
          const uint32_t k_base = smem_u32(sK + s * TB);
#pragma unroll
          for (int kk = 0; kk < 8; ++kk) {
            const uint32_t off = (kk >> 2) * HB + (kk & 3) * 32;
            mma_bf16(tmem + s * BK, desc_sw128(q_base + off), desc_sw128(k_base + off), id_s, kk > 0);
          }
          mma_commit(k_empty + s);
          mma_commit(s_full + s);
        }
        if (t >= 1) {
          const int u = t - 1, s = u & 1;
          if (!(ok = mbar_wait(p_full + s, (u >> 1) & 1, abort_flag))) break;
          if (!(ok = mbar_wait(v_full + s, (u >> 1) & 1, abort_flag))) break;
          fence_after_sync();
          const uint32_t p_base = smem_u32(sP + s * TB);
          const uint32_t v_base = smem_u32(sV + s * TB);
#pragma unroll
          for (int kk = 0; kk < 8; ++kk) {
            const uint32_t aoff = (kk >> 2) * HB + (kk & 3) * 32;
            mma_bf16(tmem + O_COL, desc_sw128(p_base + aoff), desc_sw128_mn(v_base + kk * 2048, HB, 1024), id_o,
                     (u > 0 || kk > 0) ? 1u : 0u);
          }
          mma_commit(v_empty + s);
          mma_commit(p_free + s);
          mma_commit(pv_done);
          pv_issued = u + 1;
        }
      }
      if (!ok) {
        *abort_flag = 1;
        dev_fail(j.L, DEV_TIMEOUT, 401);
      }
      if (pv_issued > 0) {
        volatile int no_abort = 0;
        mbar_wait(pv_done, (pv_issued - 1) & 1, &no_abort);
      }
    }
  } else {
    // ---------------- softmax and output: thread = query row = TMEM lane
    const int qd = warp & 3;
    const int r = qd * 32 + lane;
    const uint32_t lane_off = (uint32_t)(qd * 32) << 16;
    float mrun = -INFINITY, l = 0.f;
    bool ok = true;
    for (int t = 0; t < nt; ++t) {
      const int s = t & 1;
      const bool bank = t < nb;
      const int valid = bank ? min(BK, m - t * BK) : min(BK, W - (t - nb) * BK);
      ok = ok && __all_sync(0xffffffffu, mbar_wait(s_full + s, (t >> 1) & 1, abort_flag));
      if (!ok) break;
      fence_after_sync();
      float sv[128];
#pragma unroll
      for (int c = 0; c < 4; ++c) {
        float v[32];
        tmem_ld32(tmem + lane_off + s * BK + c * 32, v);
#pragma unroll
        for (int i = 0; i < 32; ++i) sv[c * 32 + i] = v[i];
      }
      tmem_wait_ld();
      fence_before_sync();
      __syncwarp();
      if (lane == 0) mbar_arrive(s_free + s);
      float tmax = -INFINITY;
#pragma unroll
      for (int i = 0; i < 128; ++i) {
        sv[i] = i < valid ? sv[i] * j.sl2 : -INFINITY;
        tmax = fmaxf(tmax, sv[i]);
      }
      // lazily raised running maximum; O and l are rescaled only when it moves by > 8
      const bool raise = tmax > mrun + RESCALE_LOG2;
      const float mnew = raise ? tmax : mrun;
      if (__any_sync(0xffffffffu, raise && t > 0)) {
        // O holds sum_{u < t} P_u V_u: wait for PV_{t-1}, then scale it in TMEM
        ok = ok && __all_sync(0xffffffffu, mbar_wait(pv_done, (t - 1) & 1, abort_flag));
        if (!ok) break;
        fence_after_sync();
        const float alpha = raise ? ex2(mrun - mnew) : 1.0f;
#pragma unroll
        for (int c = 0; c < 4; ++c) {
          float v[32];
          tmem_ld32(tmem + lane_off + O_COL + c * 32, v);
          tmem_wait_ld();
          uint32_t w32[32];
#pragma unroll
          for (int i = 0; i < 32; ++i) w32[i] = __float_as_uint(v[i] * alpha);
          tmem_st32(tmem + lane_off + O_COL + c * 32, w32);
        }
        tmem_wait_st();
      }
      if (raise) {
        l *= (t > 0) ? ex2(mrun - mnew) : 0.f;
        mrun = mnew;
      }
      // P_t into the shared-memory buffer s once PV_{t-2} has released it
      ok = ok && __all_sync(0xffffffffu, mbar_wait(p_free + s, ((t >> 1) & 1) ^ 1, abort_flag));
      if (!ok) break;
      uint8_t* pb = sP + s * TB;
#pragma unroll
      for (int c = 0; c < 16; ++c) {          // 16 chunks of 8 keys (16 bytes)
        float p[8];
#pragma unroll
        for (int i = 0; i < 8; ++i) {
          p[i] = ex2(sv[c * 8 + i] - mrun);
          l += p[i];
        }
        uint4 pk;
        pk.x = pack_bf16(p[0], p[1]);
        pk.y = pack_bf16(p[2], p[3]);
        pk.z = pack_bf16(p[4], p[5]);
        pk.w = pack_bf16(p[6], p[7]);
        const int panel = c >> 3, chunk = c & 7;
        *reinterpret_cast<uint4*>(pb + panel * HB + r * 128 + ((chunk ^ (r & 7)) << 4)) = pk;
      }
      asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
      fence_before_sync();
      __syncwarp();
      if (lane == 0) mbar_arrive(p_full + s);
    }
    // output row
    const int qrow = q0 + r;
    float o[128];
    if (ok && nt > 0) {
      ok = __all_sync(0xffffffffu, mbar_wait(pv_done, (nt - 1) & 1, abort_flag));
      if (ok) {
        fence_after_sync();
#pragma unroll
        for (int c = 0; c < 4; ++c) {
          float v[32];
          tmem_ld32(tmem + lane_off + O_COL + c * 32, v);
#pragma unroll
          for (int i = 0; i < 32; ++i) o[c * 32 + i] = v[i];
        }
        tmem_wait_ld();
      }
    }
    if (!ok) {
      *abort_flag = 1;
      if (lane == 0) dev_fail(j.L, DEV_TIMEOUT, 402);
    }
    const float inv = (ok && nt > 0 && l > 0.f) ? 1.0f / l : 0.f;
    if (qrow < j.Nq) {
      uint4* dst = reinterpret_cast<uint4*>(j.O + ((int64_t)h * j.Nq + qrow) * 128);
#pragma unroll
      for (int c = 0; c < 16; ++c) {
        uint4 pk;
        const float* x = o + c * 8;
        const bool z = !(ok && nt > 0);
        pk.x = pack_bf16(z ? 0.f : x[0] * inv, z ? 0.f : x[1] * inv);
        pk.y = pack_bf16(z ? 0.f : x[2] * inv, z ? 0.f : x[3] * inv);
        pk.z = pack_bf16(z ? 0.f : x[4] * inv, z ? 0.f : x[5] * inv);
        pk.w = pack_bf16(z ? 0.f : x[6] * inv, z ? 0.f : x[7] * inv);
        dst[c] = pk;
      }
    }
  }
  fence_before_sync();
  __syncthreads();
  if (warp == 1) {
    fence_after_sync();
    tmem_dealloc(tmem, TMEM_COLS);
  }
}

}  // namespace

cudaError_t tc_attn_set_smem_limits() {
  return cudaFuncSetAttribute(tc_attend, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)SMEM_BYTES);
}

cudaError_t launch_attend_tc(const Bank& b, DevLayer* L, const void* Q, int Nq, const void* Kw, const void* Vw,
                             int W, void* O, cudaStream_t s, Timer* t) {
  CUtensorMap mq, mkb, mvb, mkw, mvw;
  if (!make_map_rows(&mq, Q, Nq, b.H, BQ) || !make_map_rows(&mkb, b.k, b.M_max, b.H, BK) ||
      !make_map_rows(&mvb, b.v, b.M_max, b.H, BK))
    return cudaErrorInvalidValue;
  if (W > 0) {
    if (!make_map_rows(&mkw, Kw, W, b.H, BK) || !make_map_rows(&mvw, Vw, W, b.H, BK)) return cudaErrorInvalidValue;
  } else {
    mkw = mkb;   // never read: there are no window tiles
    mvw = mvb;
  }
  AttnJob job{b, L, Nq, W, (__nv_bfloat16*)O, 1.4426950408889634f / sqrtf(128.0f)};
  dim3 grid((Nq + BQ - 1) / BQ, b.H);
  timer_begin(t, "attend_tc", s);
  tc_attend<<<grid, THREADS, SMEM_BYTES, s>>>(mq, mkb, mvb, mkw, mvw, job);
  timer_end(t, s);
  return cudaGetLastError();
}

}  // namespace dkv
