// Bank-reading attention on the tensor cores (bf16, d = 128):
//   O = softmax(Q [K_bank ; K_win]^T / sqrt(d)) [V_bank ; V_win]        (Sec. 3.2, Fig. 2)
// over the m_h retained bank states followed by the W window states, no mask.
//
// One CTA owns 128 queries of one head.  The key range (bank tiles, then window
// tiles, 128 keys each) is split in two halves, processed concurrently by two
// softmax warpgroups that share the query tile and one MMA-issuing thread:
//   S_g = Q K^T            tcgen05.mma into TMEM (128 columns per group)
//   P_g = exp2(S_g log2(e)/sqrt(d) - m_g)   softmax threads (thread = query row);
//                          P is written back over S_g in TMEM as packed bf16
//   O_g += P_g V           tcgen05.mma with A = P_g read from TMEM, V MN-major in smem
// The running maximum m_g is raised only when a tile's maximum exceeds it by more
// than 8 (log2 units); O_g and the running sum are then rescaled in TMEM.  At the
// end the two partial results are merged exactly:
//   O = (2^(m_0 - m) O_0 + 2^(m_1 - m) O_1) / (2^(m_0 - m) l_0 + 2^(m_1 - m) l_1).
// Warps: 0 TMA producer, 1 MMA issuer, 2-5 softmax group 0, 6-9 softmax group 1.
// TMEM columns: S_0 [0,128), O_0 [128,256), S_1 [256,384), O_1 [384,512).
// The MMA-issuing thread waits once per group and tile (any wait there stalls the
// tensor pipe): p_full_g completes when the softmax has written P_g(i) AND V(i) and
// K(i + 1) have landed (the producer arms it with their bytes; K has two slots per
// group, so K(i + 1) loads while S_g(i) still reads K(i)).
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
constexpr int THREADS = 64 + 256;
constexpr uint32_t TMEM_COLS = 512;
constexpr int OFF_Q = 0;
constexpr int OFF_K = TB;               // [2 groups][2 slots]
constexpr int OFF_V = 5 * TB;           // [2 groups]
constexpr int OFF_X = 7 * TB;           // float [2 groups][2 (m, l)][BQ]
constexpr int OFF_BAR = OFF_X + 2 * 2 * BQ * 4;
constexpr size_t SMEM_BYTES = OFF_BAR + 256;   // base 1024-aligned (checked)
constexpr float RESCALE_LOG2 = 8.0f;

__device__ __forceinline__ float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// max(a, b, c) in one instruction (three-input form, sm_100 and later).
__device__ __forceinline__ float max3(float a, float b, float c) {
  float y;
  asm("max.f32 %0, %1, %2, %3;" : "=f"(y) : "f"(a), "f"(b), "f"(c));
  return y;
}

__device__ __forceinline__ uint32_t pack_bf16(float a, float b) {
  __nv_bfloat162 v = __floats2bfloat162_rn(a, b);
  return *reinterpret_cast<uint32_t*>(&v);
}

// Row maximum accumulation over 32 scores (t: eight partial maxima).
__device__ __forceinline__ void max_acc(float (&t)[8], const float (&v)[32]) {
#pragma unroll
  for (int k = 0; k < 16; ++k) t[k & 7] = max3(t[k & 7], v[2 * k], v[2 * k + 1]);
}

// Scores of the columns at or past `lim` (keys past the end of the range) become -inf:
// they do not raise the maximum and their exponentials are exactly 0.
__device__ __forceinline__ void mask_tail(float (&v)[32], int lim) {
#pragma unroll
  for (int k = 0; k < 32; ++k)
    if (k >= lim) v[k] = -INFINITY;
}

// P = 2^(s sl2 - m) over 64 scores (a: the first 32, b: the next 32) as 32 packed bf16
// pairs; lab accumulates the even and the odd columns.
__device__ __forceinline__ void exp_pack(const float (&a)[32], const float (&b)[32], float sl2, float nm,
                                         float2& lab, uint32_t (&pk)[32]) {
  const float2 sl2x2 = make_float2(sl2, sl2), nmx2 = make_float2(nm, nm);
#pragma unroll
  for (int k = 0; k < 32; ++k) {
    const float s0 = k < 16 ? a[2 * k] : b[2 * k - 32];
    const float s1 = k < 16 ? a[2 * k + 1] : b[2 * k - 31];
    const float2 x = __ffma2_rn(make_float2(s0, s1), sl2x2, nmx2);
    const float2 pp = make_float2(ex2(x.x), ex2(x.y));
    lab = __fadd2_rn(lab, pp);
    pk[k] = pack_bf16(pp.x, pp.y);
  }
}

struct AttnJob {
  Bank b;
  DevLayer* L;   // sticky error word
  int Nq;
  int W;
  __nv_bfloat16* O;
  float sl2;     // log2(e) / sqrt(d)
};

__global__ void __launch_bounds__(THREADS, 1)
    tc_attend(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmKb,
              const __grid_constant__ CUtensorMap tmVb, const __grid_constant__ CUtensorMap tmKw,
              const __grid_constant__ CUtensorMap tmVw, AttnJob j) {
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  if ((smem_u32(smem_raw) & 1023u) != 0u) {   // 128-byte-swizzled tiles need 1024-byte alignment
    if (threadIdx.x == 0) dev_fail(j.L, DEV_INCONSISTENT, 9901);
    return;
  }
  uint8_t* smem = smem_raw;
  float* xst = reinterpret_cast<float*>(smem + OFF_X);
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + OFF_BAR);
  uint64_t* q_full = bars + 0;
  uint64_t* k0_full = bars + 1;   // [2 groups] first K tile of the group
  uint64_t* k_empty = bars + 3;   // [2 groups][2 slots] S_g of the slot's tile complete
  uint64_t* v_empty = bars + 7;   // [2] PV_g complete (V slot free)
  uint64_t* s_full = bars + 9;    // [2]
  uint64_t* p_full = bars + 11;   // [2] P_g(i) written, V(i) and K(i + 1) landed
  uint64_t* pv_done = bars + 13;  // [2]
  uint32_t* tmem_holder = reinterpret_cast<uint32_t*>(bars + 15);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_holder + 1);

  const int h = blockIdx.y;
  const int q0 = blockIdx.x * BQ;
  const int m = min(max(j.b.occ[h], 0), j.b.M_max);
  const int W = j.W;
  const int nb = (m + BK - 1) / BK;            // bank tiles
  const int nt = nb + (W + BK - 1) / BK;       // all key tiles
  const int nh = (nt + 1) / 2;                 // tiles of group 0; group 1 takes the rest
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    mbar_init(q_full, 1);
    for (int g = 0; g < 2; ++g) {
      mbar_init(k0_full + g, 1);
      mbar_init(k_empty + 2 * g, 1); mbar_init(k_empty + 2 * g + 1, 1);
      mbar_init(v_empty + g, 1);
      mbar_init(s_full + g, 1);
      mbar_init(p_full + g, 4 + 1);   // four softmax warps + the producer (with bytes)
      mbar_init(pv_done + g, 1);
    }
    *abort_flag = 0;
    fence_barrier_init();
  }
  if (warp == 1) tmem_alloc(tmem_holder, TMEM_COLS);
  fence_before_sync();
  __syncthreads();
  fence_after_sync();
  const uint32_t tmem = *tmem_holder;

  auto tiles_of = [&](int g) { return g == 0 ? nh : nt - nh; };
  auto tile_index = [&](int g, int i) { return g * nh + i; };

  if (warp == 0) {
    if (lane == 0 && nt > 0) {
      // ---------------- TMA producer: Q once; per group K(0), then for each tile i the
      // bytes of V(i) and K(i + 1) on p_full_g (phase i)
      prefetch_map(&tmQ);
      mbar_arrive_expect_tx(q_full, TB);
      tma_load_3d(smem + OFF_Q, &tmQ, q_full, 0, q0, h);
      tma_load_3d(smem + OFF_Q + HB, &tmQ, q_full, 64, q0, h);
      const int n[2] = {tiles_of(0), tiles_of(1)};
      auto load_tile = [&](bool is_k, int g, int i, void* dst, uint64_t* bar) {
        const int u = tile_index(g, i);
        const bool bank = u < nb;
        const CUtensorMap* mp = is_k ? (bank ? &tmKb : &tmKw) : (bank ? &tmVb : &tmVw);
        const int row = bank ? u * BK : (u - nb) * BK;
        tma_load_3d(dst, mp, bar, 0, row, h);
        tma_load_3d(static_cast<uint8_t*>(dst) + HB, mp, bar, 64, row, h);
      };
      for (int g = 0; g < 2; ++g)
        if (n[g] > 0) {
          mbar_arrive_expect_tx(k0_full + g, TB);
          load_tile(true, g, 0, smem + OFF_K + (2 * g) * TB, k0_full + g);
        }
      int armed[2] = {0, 0};   // p_full phases armed per group
      bool ok = true;
      for (int i = 0; ok && i < n[0]; ++i) {
        for (int g = 0; g < 2 && ok; ++g) {
          if (i >= n[g]) continue;
          // PV_g(i - 1) complete: the V slot is free and p_full_g phase i - 1 is over
          if (i > 0 && !(ok = mbar_wait(v_empty + g, (i - 1) & 1, abort_flag))) break;
          const bool knext = i + 1 < n[g];
          // S_g(i - 1) complete: K slot (i + 1) & 1 is free
          if (knext && i > 0 && !(ok = mbar_wait(k_empty + 2 * g + ((i + 1) & 1), ((i - 1) >> 1) & 1, abort_flag)))
            break;
          mbar_arrive_expect_tx(p_full + g, knext ? 2 * TB : TB);
          load_tile(false, g, i, smem + OFF_V + g * TB, p_full + g);
          if (knext) load_tile(true, g, i + 1, smem + OFF_K + (2 * g + ((i + 1) & 1)) * TB, p_full + g);
          armed[g] = i + 1;
        }
      }
      if (!ok) {
        *abort_flag = 1;
        dev_fail(j.L, DEV_TIMEOUT, 400);
      }
      // never leave with copies in flight: earlier phases completed before this thread
      // armed the next one; the last armed phase also needs the softmax, which an
      // aborted CTA may never give: then wait a fixed 50 us, far longer than a copy takes
      volatile int no_abort = 0;
      mbar_wait(q_full, 0, &no_abort);
      bool drained = true;
      for (int g = 0; g < 2; ++g) {
        if (n[g] > 0) mbar_wait(k0_full + g, 0, &no_abort);
        if (armed[g] > 0) drained = drained && mbar_wait(p_full + g, (armed[g] - 1) & 1, abort_flag);
      }
      if (!drained) {
        const uint64_t t0 = globaltimer_ns();
        while (globaltimer_ns() - t0 < 50000ull) {
        }
      }
    }
  } else if (warp == 1) {
    if (lane == 0 && nt > 0) {
      // ---------------- MMA issuer.  Per group: S(0), then for each tile i:
      // PV(i) once P(i) is in TMEM, then S(i+1) (which overwrites P(i) after PV(i) read it).
      constexpr uint32_t id_s = idesc_bf16(BQ, BK);
      constexpr uint32_t id_o = idesc_bf16(BQ, 128, /*b_mn_major=*/true);
      const uint32_t q_base = smem_u32(smem + OFF_Q);
      const int n[2] = {tiles_of(0), tiles_of(1)};
      bool ok = mbar_wait(q_full, 0, abort_flag);
      int pv_issued[2] = {0, 0};
      // S_g(i): its K tile has landed (K(0): k0_full; K(i + 1): with p_full_g phase i)
      const uint64_t qd = desc_sw128(q_base), kd0 = desc_sw128(smem_u32(smem + OFF_K));
      const uint64_t vd0 = desc_sw128_mn(smem_u32(smem + OFF_V), HB, 1024);
      auto issue_s = [&](int g, int i) {
        const uint64_t kd = desc_add(kd0, (2 * g + (i & 1)) * TB);
        const uint32_t sc = tmem + g * 256;
#pragma unroll
        for (int kk = 0; kk < 8; ++kk) {
          const uint32_t off = (kk >> 2) * HB + (kk & 3) * 32;
          mma_bf16(sc, desc_add(qd, off), desc_add(kd, off), id_s, kk > 0);
        }
        mma_commit(k_empty + 2 * g + (i & 1));
        mma_commit(s_full + g);
      };
      auto issue_pv = [&](int g, int i) -> bool {
        if (!mbar_wait(p_full + g, i & 1, abort_flag)) return false;   // the one wait
        fence_after_sync();
        const uint64_t vd = desc_add(vd0, g * TB);
        const uint32_t pc = tmem + g * 256;          // P: packed bf16 pairs over S columns [0, 64)
        const uint32_t oc = tmem + g * 256 + 128;
#pragma unroll
        for (int kk = 0; kk < 8; ++kk)
          mma_bf16_ts(oc, pc + kk * 8, desc_add(vd, kk * 2048), id_o, (i > 0 || kk > 0) ? 1u : 0u);
        mma_commit(v_empty + g);
        mma_commit(pv_done + g);
        pv_issued[g] = i + 1;
        return true;
      };
      for (int g = 0; g < 2 && ok; ++g)
        if (n[g] > 0) {
          if ((ok = mbar_wait(k0_full + g, 0, abort_flag))) {
            fence_after_sync();
            issue_s(g, 0);
          }
        }
      for (int i = 0; ok && i < n[0]; ++i) {
        for (int g = 0; g < 2 && ok; ++g) {
          if (i >= n[g]) continue;
          ok = issue_pv(g, i);
          if (ok && i + 1 < n[g]) issue_s(g, i + 1);
        }
      }
      if (!ok) {
        *abort_flag = 1;
        dev_fail(j.L, DEV_TIMEOUT, 401);
      }
      volatile int no_abort = 0;
      for (int g = 0; g < 2; ++g)
        if (pv_issued[g] > 0) mbar_wait(pv_done + g, (pv_issued[g] - 1) & 1, &no_abort);
    }
  } else {
    // ---------------- softmax group g, thread = query row = TMEM lane
    const int g = (warp - 2) >> 2;
    const int qd = warp & 3;
    const int r = qd * 32 + lane;
    const uint32_t lane_off = (uint32_t)(qd * 32) << 16;
    const uint32_t sc = tmem + lane_off + g * 256;     // S_g (and P_g)
    const uint32_t oc = sc + 128;                      // O_g
    const int ng = tiles_of(g);
    float mrun = -INFINITY, l = 0.f;
    bool ok = true;
    for (int i = 0; i < ng; ++i) {
      const int u = tile_index(g, i);
      const bool bank = u < nb;
      const int valid = bank ? min(BK, m - u * BK) : min(BK, W - (u - nb) * BK);
      ok = ok && __all_sync(0xffffffffu, mbar_wait(s_full + g, i & 1, abort_flag));
      if (!ok) break;
      fence_after_sync();
      // the whole row of S_g (128 scores) in registers: four loads, one wait
      float s0[32], s1[32], s2[32], s3[32];
      tmem_ld32(sc, s0);
      tmem_ld32(sc + 32, s1);
      tmem_ld32(sc + 64, s2);
      tmem_ld32(sc + 96, s3);
      tmem_wait_ld();
      if (valid < BK) {   // partial last tile of the bank or of the window
        mask_tail(s0, valid); mask_tail(s1, valid - 32); mask_tail(s2, valid - 64); mask_tail(s3, valid - 96);
      }
      // row maximum of the raw scores
      float tmax;
      {
        float t[8];
#pragma unroll
        for (int k = 0; k < 8; ++k) t[k] = -INFINITY;
        max_acc(t, s0); max_acc(t, s1); max_acc(t, s2); max_acc(t, s3);
        tmax = fmaxf(fmaxf(fmaxf(t[0], t[1]), fmaxf(t[2], t[3])), fmaxf(fmaxf(t[4], t[5]), fmaxf(t[6], t[7])));
      }
      tmax *= j.sl2;
      // lazily raised running maximum.  S_g(i) complete implies PV_g(i-1) complete
      // (one thread issues both, in order), so O_g is idle here.
      const bool raise = tmax > mrun + RESCALE_LOG2;
      const float mnew = raise ? tmax : mrun;
      const float mprev = mrun;
      if (raise) {
        l *= (i > 0) ? ex2(mrun - mnew) : 0.f;
        mrun = mnew;
      }
      // P_g = 2^(s log2(e)/sqrt(d) - m) as packed bf16 pairs over the first 64 columns of S_g
      const float nm = -mrun;
      float2 lab = make_float2(0.f, 0.f);     // running sums of the even and odd columns
      {
        uint32_t pk[32];
        exp_pack(s0, s1, j.sl2, nm, lab, pk);
        tmem_st32(sc, pk);
        exp_pack(s2, s3, j.sl2, nm, lab, pk);
        tmem_st32(sc + 32, pk);
      }
      // O_g rescale: after the P stores (S is dead), before PV(i) is released
      if (__any_sync(0xffffffffu, raise && i > 0)) {
        const float alpha = raise ? ex2(mprev - mnew) : 1.0f;
#pragma unroll
        for (int c = 0; c < 4; ++c) {
          float v[32];
          tmem_ld32(oc + c * 32, v);
          tmem_wait_ld();
          uint32_t w32[32];
#pragma unroll
          for (int k = 0; k < 16; ++k) {
            const float2 y = __fmul2_rn(make_float2(v[2 * k], v[2 * k + 1]), make_float2(alpha, alpha));
            w32[2 * k] = __float_as_uint(y.x);
            w32[2 * k + 1] = __float_as_uint(y.y);
          }
          tmem_st32(oc + c * 32, w32);
        }
      }
      l += lab.x + lab.y;
      tmem_wait_st();
      fence_before_sync();
      __syncwarp();
      if (lane == 0) mbar_arrive(p_full + g);
    }
    // ---- merge the two groups' partial softmax results
    if (ok && ng > 0) ok = __all_sync(0xffffffffu, mbar_wait(pv_done + g, (ng - 1) & 1, abort_flag));
    if (!ok) {
      *abort_flag = 1;
      if (lane == 0) dev_fail(j.L, DEV_TIMEOUT, 402);
    }
    xst[(g * 2 + 0) * BQ + r] = ng > 0 && ok ? mrun : -INFINITY;
    xst[(g * 2 + 1) * BQ + r] = ng > 0 && ok ? l : 0.f;
    named_bar(1 + qd, 64);   // the two warps (one per group) of this TMEM lane quarter
    const float m0 = xst[0 * BQ + r], l0 = xst[1 * BQ + r];
    const float m1 = xst[2 * BQ + r], l1 = xst[3 * BQ + r];
    const float mm = fmaxf(m0, m1);
    const float a0 = m0 == -INFINITY ? 0.f : ex2(m0 - mm);
    const float a1 = m1 == -INFINITY ? 0.f : ex2(m1 - mm);
    const float den = fmaf(a1, l1, a0 * l0);
    const float inv = den > 0.f ? 1.0f / den : 0.f;
    const float c0 = a0 * inv, c1 = a1 * inv;
    // the merge reads the other group's O too: observe its last PV completion as well
    {
      const int no = tiles_of(g ^ 1);
      if (ok && no > 0) ok = __all_sync(0xffffffffu, mbar_wait(pv_done + (g ^ 1), (no - 1) & 1, abort_flag));
    }
    fence_after_sync();
    // group g writes output columns [64 g, 64 g + 64) of this row from both O_0 and O_1
    const int qrow = q0 + r;
    const uint32_t o0 = tmem + lane_off + 128 + g * 64;
    const uint32_t o1 = tmem + lane_off + 256 + 128 + g * 64;
    const bool has0 = ok && tiles_of(0) > 0 && c0 != 0.f, has1 = ok && tiles_of(1) > 0 && c1 != 0.f;
#pragma unroll
    for (int c = 0; c < 2; ++c) {
      float x0[32], x1[32];
      tmem_ld32(o0 + c * 32, x0);
      tmem_ld32(o1 + c * 32, x1);
      tmem_wait_ld();
      if (qrow < j.Nq) {
        uint4* dst = reinterpret_cast<uint4*>(j.O + ((int64_t)h * j.Nq + qrow) * 128 + g * 64 + c * 32);
#pragma unroll
        for (int k = 0; k < 4; ++k) {
          float y[8];
#pragma unroll
          for (int e = 0; e < 8; ++e) {
            const float t0 = has0 ? x0[k * 8 + e] * c0 : 0.f;
            y[e] = has1 ? fmaf(x1[k * 8 + e], c1, t0) : t0;
          }
          uint4 pk;
          pk.x = pack_bf16(y[0], y[1]);
          pk.y = pack_bf16(y[2], y[3]);
          pk.z = pack_bf16(y[4], y[5]);
          pk.w = pack_bf16(y[6], y[7]);
          dst[k] = pk;
        }
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

// ---------------------------------------------------------------------------------
// Two query tiles per CTA.  One CTA owns 256 queries of one head as two 128-query
// tiles Q_0, Q_1 that read every key tile together: each K and V tile crosses from L2
// into shared memory once per 256 queries instead of once per 128, which halves the
// L2 -> shared-memory traffic per MMA (one K/V tile per 128 queries needs about as many
// bytes per cycle as an SM can take from L2 while its tensor pipe is busy).  Softmax
// group g (four warps, thread = query row) owns Q_g over the whole key range, so no
// merge is needed at the end.  TMEM columns as above: S_g, O_g for g = 0, 1.
// Shared memory: Q_0, Q_1, two K slots, three V slots (224 KiB).
// MMA issuer, per tile i: [wait pf0(i)] PV_0(i), S_0(i+1); [wait pf1(i)] PV_1(i), S_1(i+1).
// pf0 (one barrier per tile parity, so the producer can arm tile i + 1 while tile i is
// open) completes when softmax group 0 has written P_0(i) and V(i), K(i+1) have landed;
// pf1 when group 1 has written P_1(i).  With a single valid query tile (the last 128
// queries of a head) group 1 takes no part.
constexpr int OFF2_Q = 0;               // [2] query tiles
constexpr int OFF2_K = 2 * TB;          // [2] key slots
constexpr int OFF2_V = 4 * TB;          // [3] value slots
constexpr int OFF2_BAR = 7 * TB;
constexpr size_t SMEM2_BYTES = OFF2_BAR + 256;   // base 1024-aligned (checked)
static_assert(SMEM2_BYTES <= 227 * 1024, "shared memory per CTA");

__global__ void __launch_bounds__(THREADS, 1)
    tc_attend2(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmKb,
               const __grid_constant__ CUtensorMap tmVb, const __grid_constant__ CUtensorMap tmKw,
               const __grid_constant__ CUtensorMap tmVw, AttnJob j) {
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  if ((smem_u32(smem_raw) & 1023u) != 0u) {
    if (threadIdx.x == 0) dev_fail(j.L, DEV_INCONSISTENT, 9902);
    return;
  }
  uint8_t* smem = smem_raw;
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + OFF2_BAR);
  uint64_t* q_full = bars + 0;
  uint64_t* k0_full = bars + 1;
  uint64_t* pf0 = bars + 2;       // [2] by tile parity
  uint64_t* pf1 = bars + 4;
  uint64_t* k_empty = bars + 5;   // [2] S_0(i), S_1(i) complete: K slot i & 1 free
  uint64_t* v_empty = bars + 7;   // [3] PV_0(i), PV_1(i) complete: V slot i % 3 free
  uint64_t* s_full = bars + 10;   // [2] S_g(i) complete
  uint64_t* pv_done = bars + 12;  // [2] PV_g(i) complete
  uint32_t* tmem_holder = reinterpret_cast<uint32_t*>(bars + 14);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_holder + 1);

  const int h = blockIdx.y;
  const int q0 = blockIdx.x * 2 * BQ;
  const int G = q0 + BQ < j.Nq ? 2 : 1;         // query tiles with at least one valid query
  const int m = min(max(j.b.occ[h], 0), j.b.M_max);
  const int W = j.W;
  const int nb = (m + BK - 1) / BK;
  const int nt = nb + (W + BK - 1) / BK;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    mbar_init(q_full, 1);
    mbar_init(k0_full, 1);
    mbar_init(pf0 + 0, 4 + 1);   // four softmax warps + the producer (with bytes)
    mbar_init(pf0 + 1, 4 + 1);
    mbar_init(pf1, 4);
    for (int s = 0; s < 2; ++s) mbar_init(k_empty + s, 1);
    for (int s = 0; s < 3; ++s) mbar_init(v_empty + s, 1);
    for (int g = 0; g < 2; ++g) {
      mbar_init(s_full + g, 1);
      mbar_init(pv_done + g, 1);
    }
    *abort_flag = 0;
    fence_barrier_init();
  }
  if (warp == 1) tmem_alloc(tmem_holder, TMEM_COLS);
  fence_before_sync();
  __syncthreads();
  fence_after_sync();
  const uint32_t tmem = *tmem_holder;

  auto load_tile = [&](bool is_k, int u, void* dst, uint64_t* bar) {
    const bool bank = u < nb;
    const CUtensorMap* mp = is_k ? (bank ? &tmKb : &tmKw) : (bank ? &tmVb : &tmVw);
    const int row = bank ? u * BK : (u - nb) * BK;
    tma_load_3d(dst, mp, bar, 0, row, h);
    tma_load_3d(static_cast<uint8_t*>(dst) + HB, mp, bar, 64, row, h);
  };

  if (warp == 0) {
    if (lane == 0 && nt > 0) {
      // ---------------- TMA producer
      prefetch_map(&tmQ);
      mbar_arrive_expect_tx(q_full, G * TB);
      for (int g = 0; g < G; ++g) {
        tma_load_3d(smem + OFF2_Q + g * TB, &tmQ, q_full, 0, q0 + g * BQ, h);
        tma_load_3d(smem + OFF2_Q + g * TB + HB, &tmQ, q_full, 64, q0 + g * BQ, h);
      }
      mbar_arrive_expect_tx(k0_full, TB);
      load_tile(true, 0, smem + OFF2_K, k0_full);
      int armed = 0;
      bool ok = true;
      for (int i = 0; i < nt; ++i) {
        // pf0 of this parity: the phase of tile i - 2 is over
        if (i >= 2 && !(ok = mbar_wait(pf0 + (i & 1), ((i - 2) >> 1) & 1, abort_flag))) break;
        // V slot i % 3: the P.V products of tile i - 3 are complete
        if (i >= 3 && !(ok = mbar_wait(v_empty + i % 3, ((i - 3) / 3) & 1, abort_flag))) break;
        const bool knext = i + 1 < nt;
        // K slot (i + 1) & 1: the score products of tile i - 1 are complete
        if (knext && i >= 1 && !(ok = mbar_wait(k_empty + ((i + 1) & 1), ((i - 1) >> 1) & 1, abort_flag))) break;
        mbar_arrive_expect_tx(pf0 + (i & 1), knext ? 2 * TB : TB);
        load_tile(false, i, smem + OFF2_V + (i % 3) * TB, pf0 + (i & 1));
        if (knext) load_tile(true, i + 1, smem + OFF2_K + ((i + 1) & 1) * TB, pf0 + (i & 1));
        armed = i + 1;
      }
      if (!ok) {
        *abort_flag = 1;
        dev_fail(j.L, DEV_TIMEOUT, 410);
      }
      // never leave with copies in flight (see tc_attend)
      volatile int no_abort = 0;
      mbar_wait(q_full, 0, &no_abort);
      mbar_wait(k0_full, 0, &no_abort);
      bool drained = true;
      for (int i = armed > 2 ? armed - 2 : 0; i < armed; ++i)
        drained = drained && mbar_wait(pf0 + (i & 1), (i >> 1) & 1, abort_flag);
      if (!drained) {
        const uint64_t t0 = globaltimer_ns();
        while (globaltimer_ns() - t0 < 50000ull) {
        }
      }
    }
  } else if (warp == 1) {
    if (lane == 0 && nt > 0) {
      // ---------------- MMA issuer
      constexpr uint32_t id_s = idesc_bf16(BQ, BK);
      constexpr uint32_t id_o = idesc_bf16(BQ, 128, /*b_mn_major=*/true);
      bool ok = mbar_wait(q_full, 0, abort_flag) && mbar_wait(k0_full, 0, abort_flag);
      int pv_issued = 0;
      // every operand's descriptor once; the k-steps' by one add each (desc_add): the
      // issuing thread's time per MMA is what paces the tensor pipe here
      const uint64_t qd0 = desc_sw128(smem_u32(smem + OFF2_Q)), qd1 = desc_sw128(smem_u32(smem + OFF2_Q + TB));
      const uint64_t kd0 = desc_sw128(smem_u32(smem + OFF2_K));
      const uint64_t vd0 = desc_sw128_mn(smem_u32(smem + OFF2_V), HB, 1024);
      auto issue_s = [&](int g, int i) {
        const uint64_t qd = g ? qd1 : qd0;
        const uint64_t kd = desc_add(kd0, (i & 1) * TB);
        const uint32_t sc = tmem + g * 256;
#pragma unroll
        for (int kk = 0; kk < 8; ++kk) {
          const uint32_t off = (kk >> 2) * HB + (kk & 3) * 32;
          mma_bf16(sc, desc_add(qd, off), desc_add(kd, off), id_s, kk > 0);
        }
        mma_commit(s_full + g);
        if (g == G - 1) mma_commit(k_empty + (i & 1));
      };
      auto issue_pv = [&](int g, int i) {
        const uint64_t vd = desc_add(vd0, (i % 3) * TB);
        const uint32_t pc = tmem + g * 256;
        const uint32_t oc = tmem + g * 256 + 128;
#pragma unroll
        for (int kk = 0; kk < 8; ++kk)
          mma_bf16_ts(oc, pc + kk * 8, desc_add(vd, kk * 2048), id_o, (i > 0 || kk > 0) ? 1u : 0u);
        mma_commit(pv_done + g);
        if (g == G - 1) mma_commit(v_empty + i % 3);
      };
      if (ok) {
        fence_after_sync();
        for (int g = 0; g < G; ++g) issue_s(g, 0);
      }
      for (int i = 0; ok && i < nt; ++i) {
        // the one wait per group and tile
        if (!(ok = mbar_wait(pf0 + (i & 1), (i >> 1) & 1, abort_flag))) break;
        fence_after_sync();
        issue_pv(0, i);
        if (i + 1 < nt) issue_s(0, i + 1);
        if (G == 2) {
          if (!(ok = mbar_wait(pf1, i & 1, abort_flag))) break;
          fence_after_sync();
          issue_pv(1, i);
          if (i + 1 < nt) issue_s(1, i + 1);
        }
        pv_issued = i + 1;
      }
      if (!ok) {
        *abort_flag = 1;
        dev_fail(j.L, DEV_TIMEOUT, 411);
      }
      // every issued MMA complete before TMEM is freed (commits track all earlier MMAs)
      volatile int no_abort = 0;
      if (pv_issued > 0) mbar_wait(pv_done + 0, (pv_issued - 1) & 1, &no_abort);
      if (G == 2 && pv_issued > 0) mbar_wait(pv_done + 1, (pv_issued - 1) & 1, &no_abort);
    }
  } else {
    // ---------------- softmax group g over query tile g, thread = query row = TMEM lane
    const int g = (warp - 2) >> 2;
    const int qd = warp & 3;
    const int r = qd * 32 + lane;
    const uint32_t lane_off = (uint32_t)(qd * 32) << 16;
    const uint32_t sc = tmem + lane_off + g * 256;
    const uint32_t oc = sc + 128;
    const int ng = g < G ? nt : 0;
    float mrun = -INFINITY, l = 0.f;
    bool ok = true;
    for (int i = 0; i < ng; ++i) {
      const bool bank = i < nb;
      const int valid = bank ? min(BK, m - i * BK) : min(BK, W - (i - nb) * BK);
      ok = ok && __all_sync(0xffffffffu, mbar_wait(s_full + g, i & 1, abort_flag));
      if (!ok) break;
      fence_after_sync();
      float s0[32], s1[32], s2[32], s3[32];
      tmem_ld32(sc, s0);
      tmem_ld32(sc + 32, s1);
      tmem_ld32(sc + 64, s2);
      tmem_ld32(sc + 96, s3);
      tmem_wait_ld();
      if (valid < BK) {
        mask_tail(s0, valid); mask_tail(s1, valid - 32); mask_tail(s2, valid - 64); mask_tail(s3, valid - 96);
      }
      float tmax;
      {
        float t[8];
#pragma unroll
        for (int k = 0; k < 8; ++k) t[k] = -INFINITY;
        max_acc(t, s0); max_acc(t, s1); max_acc(t, s2); max_acc(t, s3);
        tmax = fmaxf(fmaxf(fmaxf(t[0], t[1]), fmaxf(t[2], t[3])), fmaxf(fmaxf(t[4], t[5]), fmaxf(t[6], t[7])));
      }
      tmax *= j.sl2;
      // S_g(i) complete implies PV_g(i - 1) complete (issued earlier by the same thread)
      const bool raise = tmax > mrun + RESCALE_LOG2;
      const float mnew = raise ? tmax : mrun;
      const float mprev = mrun;
      if (raise) {
        l *= (i > 0) ? ex2(mrun - mnew) : 0.f;
        mrun = mnew;
      }
      const float nm = -mrun;
      float2 lab = make_float2(0.f, 0.f);
      {
        uint32_t pk[32];
        exp_pack(s0, s1, j.sl2, nm, lab, pk);
        tmem_st32(sc, pk);
        exp_pack(s2, s3, j.sl2, nm, lab, pk);
        tmem_st32(sc + 32, pk);
      }
      if (__any_sync(0xffffffffu, raise && i > 0)) {
        const float alpha = raise ? ex2(mprev - mnew) : 1.0f;
#pragma unroll
        for (int c = 0; c < 4; ++c) {
          float v[32];
          tmem_ld32(oc + c * 32, v);
          tmem_wait_ld();
          uint32_t w32[32];
#pragma unroll
          for (int k = 0; k < 16; ++k) {
            const float2 y = __fmul2_rn(make_float2(v[2 * k], v[2 * k + 1]), make_float2(alpha, alpha));
            w32[2 * k] = __float_as_uint(y.x);
            w32[2 * k + 1] = __float_as_uint(y.y);
          }
          tmem_st32(oc + c * 32, w32);
        }
      }
      l += lab.x + lab.y;
      tmem_wait_st();
      fence_before_sync();
      __syncwarp();
      if (lane == 0) mbar_arrive(g == 0 ? pf0 + (i & 1) : pf1);
    }
    if (ok && ng > 0) ok = __all_sync(0xffffffffu, mbar_wait(pv_done + g, (ng - 1) & 1, abort_flag));
    if (!ok) {
      *abort_flag = 1;
      if (lane == 0) dev_fail(j.L, DEV_TIMEOUT, 412);
    }
    fence_after_sync();
    const int qrow = q0 + g * BQ + r;
    const float inv = ok && ng > 0 && l > 0.f ? 1.0f / l : 0.f;
#pragma unroll
    for (int c = 0; c < 4; ++c) {
      float x[32];
      if (ng > 0) {   // warp-uniform
        tmem_ld32(oc + c * 32, x);
        tmem_wait_ld();
      }
      if (g < G && qrow < j.Nq) {
        uint4* dst = reinterpret_cast<uint4*>(j.O + ((int64_t)h * j.Nq + qrow) * 128 + c * 32);
#pragma unroll
        for (int k = 0; k < 4; ++k) {
          float y[8];
#pragma unroll
          for (int e = 0; e < 8; ++e) y[e] = ng > 0 ? x[k * 8 + e] * inv : 0.f;
          uint4 pk;
          pk.x = pack_bf16(y[0], y[1]);
          pk.y = pack_bf16(y[2], y[3]);
          pk.z = pack_bf16(y[4], y[5]);
          pk.w = pack_bf16(y[6], y[7]);
          dst[k] = pk;
        }
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
  cudaError_t e = cudaFuncSetAttribute(tc_attend, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)SMEM_BYTES);
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(tc_attend2, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)SMEM2_BYTES);
  return e;
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
  // two query tiles per CTA whenever that still gives every SM at least two CTAs (the
  // key-split kernel keeps small grids, e.g. one layer of 12 heads, in fewer waves)
  static int n_sm = 0;
  if (n_sm == 0) {
    int dev = 0, v = 0;
    if (cudaGetDevice(&dev) == cudaSuccess &&
        cudaDeviceGetAttribute(&v, cudaDevAttrMultiProcessorCount, dev) == cudaSuccess)
      n_sm = v;
  }
  const int64_t ctas2 = (int64_t)((Nq + 2 * BQ - 1) / (2 * BQ)) * b.H;
  timer_begin(t, "attend_tc", s);
  if (n_sm > 0 && ctas2 >= 2 * (int64_t)n_sm) {
    dim3 grid((Nq + 2 * BQ - 1) / (2 * BQ), b.H);
    tc_attend2<<<grid, THREADS, SMEM2_BYTES, s>>>(mq, mkb, mvb, mkw, mvw, job);
  } else {
    dim3 grid((Nq + BQ - 1) / BQ, b.H);
    tc_attend<<<grid, THREADS, SMEM_BYTES, s>>>(mq, mkb, mvb, mkw, mvw, job);
  }
  timer_end(t, s);
  return cudaGetLastError();
}

}  // namespace dkv
