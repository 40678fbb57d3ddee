// Tensor-core (tcgen05) pair passes of the bank update, bf16 keys, d = 128.
//
// Every pass contracts a tile of 128 "row" keys against a run of "column" keys:
//   acc[i][j] = k_i . k_j                       (tcgen05.mma, bf16 in, fp32 in TMEM)
//   u = eps + (|k_i|^2 + |k_j|^2 - 2 acc) / sigma^2,  w = u^-p     (Eq. 2, fp32 epilogue)
// and folds w into a per-row quantity in the epilogue, so no row-by-column matrix
// ever reaches global memory (App. C "Decision granularity versus computational
// tiling"):
//   SCORE    rows = candidates, cols = bank:         s(x) = (1/m) sum_i w / b_i   (Eq. 6)
//   CROSS    rows = bank, cols = candidates in pi order: running rho~_i(r) (Eq. C.2),
//            first r with rho~ >= tau b_i (Eqs. 8-9), snapshots every 128 columns
//   PROJECT  rows = bank, cols = pi-ordered candidates [128 floor(r/128), r):
//            rho~_i(r) resumed from the snapshot (same tiles, same arithmetic)
//   SUB      rows = survivors, cols = evicted: rho_i = rho~_i - sum_R w     (Eq. C.4)
//   NEWBASE  rows = admitted, cols = final bank (self excluded by index):
//            rho_x = Phi(x), b_x = max(rho_x, delta)                 (Eq. 5 / C.4)
//
// CTA layout (192 threads, 2 CTAs per SM): warp 0 issues TMA (row tile once, column
// tiles through a 2-stage ring), warp 1 issues tcgen05.mma into two 128-column TMEM
// accumulators, warps 2-5 are the epilogue (thread = row = TMEM lane).
#include "dkv_internal.h"
#include "tc_ptx.cuh"

#include <climits>
#include <mutex>

namespace dkv {

namespace {

using namespace tc;

enum TMode { TM_SCORE = 0, TM_CROSS = 1, TM_PROJECT = 2, TM_SUB = 3, TM_NEWBASE = 4 };

constexpr int BM = 128;          // rows per CTA (TMEM lanes)
constexpr int BN = 128;          // columns per tile
constexpr int TILE_BYTES = BM * 128 * 2;   // 128 rows x 128 bf16
constexpr int HALF_BYTES = TILE_BYTES / 2; // one 64-column swizzle panel
constexpr int STAGES = 2;
constexpr int THREADS = 192;
constexpr uint32_t TMEM_COLS = 256;        // two 128-column accumulators
constexpr size_t SMEM_BYTES = 1024 /*align*/ + TILE_BYTES * (1 + STAGES) + 2 * 2 * BN * 4 /*meta*/ + 256;

struct TcJob {
  Bank b;
  Ws w;
  KParams kp;
  const float* rnorm;   // row key norms, head stride rn_hs
  int64_t rn_hs;
};

__device__ __forceinline__ void job_range(int MODE, const DevHead& hd, const DevLayer& L, int& nrows, int& c0,
                                          int& c1) {
  nrows = 0; c0 = 0; c1 = 0;
  if (MODE == TM_SCORE) { nrows = hd.empty ? 0 : L.N; c1 = hd.m_old; }
  if (MODE == TM_CROSS) { nrows = hd.empty ? 0 : hd.m_old; c1 = L.rmax; }
  if (MODE == TM_PROJECT) { nrows = hd.empty ? 0 : hd.m_old; c0 = (hd.r / SNAP) * SNAP; c1 = hd.r; }
  if (MODE == TM_SUB) { nrows = hd.empty ? 0 : hd.m_old - hd.e; c1 = hd.e; }
  if (MODE == TM_NEWBASE) { nrows = hd.r; c1 = hd.m_new; }
}

template <int MODE>
__global__ void __launch_bounds__(THREADS, 2)
    tc_pairs(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB, TcJob j) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);
  uint8_t* sA = smem;
  uint8_t* sB = smem + TILE_BYTES;
  float* meta = reinterpret_cast<float*>(smem + TILE_BYTES * (1 + STAGES));   // [2 buf][2][BN]
  uint64_t* bars = reinterpret_cast<uint64_t*>(meta + 2 * 2 * BN);
  uint64_t* bar_a = bars + 0;
  uint64_t* bar_full = bars + 1;    // [STAGES]
  uint64_t* bar_empty = bars + 3;   // [STAGES]
  uint64_t* bar_accf = bars + 5;    // [2]
  uint64_t* bar_acce = bars + 7;    // [2]
  uint32_t* tmem_holder = reinterpret_cast<uint32_t*>(bars + 9);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_holder + 1);

  const int h = blockIdx.y;
  const DevHead hd = j.w.hd[h];
  const DevLayer L = *j.w.L;
  int nrows, c0, c1;
  job_range(MODE, hd, L, nrows, c0, c1);
  const int row0 = blockIdx.x * BM;
  if (row0 >= nrows) return;                      // uniform: before any barrier or TMEM use
  const int ntiles = c1 > c0 ? (c1 - c0 + BN - 1) / BN : 0;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    mbar_init(bar_a, 1);
    for (int s = 0; s < STAGES; ++s) { mbar_init(bar_full + s, 1); mbar_init(bar_empty + s, 1); }
    for (int b = 0; b < 2; ++b) { mbar_init(bar_accf + b, 1); mbar_init(bar_acce + b, 4); }
    *abort_flag = 0;
    fence_barrier_init();
  }
  if (warp == 1) tmem_alloc(tmem_holder, TMEM_COLS);
  fence_before_sync();
  __syncthreads();
  fence_after_sync();
  const uint32_t tmem = *tmem_holder;

  if (warp == 0) {
    if (lane == 0 && ntiles > 0) {
      // ---------------- TMA producer
      prefetch_map(&tmA);
      prefetch_map(&tmB);
      mbar_arrive_expect_tx(bar_a, TILE_BYTES);
      tma_load_3d(sA, &tmA, bar_a, 0, row0, h);
      tma_load_3d(sA + HALF_BYTES, &tmA, bar_a, 64, row0, h);
      int issued = 0;
      for (int t = 0; t < ntiles; ++t) {
        const int s = t % STAGES;
        const uint32_t ph = (t / STAGES) & 1;
        if (!mbar_wait(bar_empty + s, ph ^ 1, abort_flag)) break;
        mbar_arrive_expect_tx(bar_full + s, TILE_BYTES);
        const int col = c0 + t * BN;
        tma_load_3d(sB + s * TILE_BYTES, &tmB, bar_full + s, 0, col, h);
        tma_load_3d(sB + s * TILE_BYTES + HALF_BYTES, &tmB, bar_full + s, 64, col, h);
        issued = t + 1;
      }
      if (issued < ntiles) {
        *abort_flag = 1;
        dev_fail(j.w.L, DEV_TIMEOUT, 100 + MODE);
      }
      // never leave with copies in flight: wait (bounded) for the last loads issued
      volatile int no_abort = 0;
      mbar_wait(bar_a, 0, &no_abort);
      for (int t = issued > STAGES ? issued - STAGES : 0; t < issued; ++t)
        mbar_wait(bar_full + (t % STAGES), (t / STAGES) & 1, &no_abort);
    }
  } else if (warp == 1) {
    if (lane == 0 && ntiles > 0) {
      // ---------------- MMA issuer
      constexpr uint32_t idesc = idesc_bf16(BM, BN);
      bool ok = mbar_wait(bar_a, 0, abort_flag);
      const uint32_t a_base = smem_u32(sA);
      int done = 0;
      for (int t = 0; ok && t < ntiles; ++t) {
        const int s = t % STAGES;
        const int b = t & 1;
        if (!mbar_wait(bar_full + s, (t / STAGES) & 1, abort_flag)) { ok = false; break; }
        if (!mbar_wait(bar_acce + b, ((t >> 1) & 1) ^ 1, abort_flag)) { ok = false; break; }
        fence_after_sync();
        const uint32_t b_base = smem_u32(sB + s * TILE_BYTES);
#pragma unroll
        for (int kk = 0; kk < 8; ++kk) {
          const uint32_t koff = (kk >> 2) * HALF_BYTES + (kk & 3) * 32;
          mma_bf16(tmem + b * BN, desc_sw128(a_base + koff), desc_sw128(b_base + koff), idesc, kk > 0);
        }
        mma_commit(bar_empty + s);
        mma_commit(bar_accf + b);
        done = t + 1;
      }
      if (!ok) {
        *abort_flag = 1;
        dev_fail(j.w.L, DEV_TIMEOUT, 200 + MODE);
      }
      // all issued MMAs must be complete before TMEM is freed
      if (done > 0) {
        volatile int no_abort = 0;
        mbar_wait(bar_accf + ((done - 1) & 1), ((done - 1) >> 1) & 1, &no_abort);
      }
    }
  } else {
    // ---------------- epilogue: one thread per row (TMEM lane)
    const int q = warp & 3;                       // TMEM lane quarter accessible to this warp
    const int r_local = q * 32 + lane;
    const int row = row0 + r_local;
    const bool active = row < nrows;
    const int et = threadIdx.x - 64;              // 0..127 among the epilogue threads
    const int64_t bh = (int64_t)h * j.b.M_max;
    const KParams kp = j.kp;
    const float k2 = -2.0f * kp.inv_s2;
    // per-row state
    float cr = kp.eps, S = 0.f, acc = 0.f, thr = 0.f;
    int cross = INT_MAX, self = -1, slot = row;
    float* snap_row = nullptr;
    if (active) {
      cr = fmaf(j.rnorm[(int64_t)h * j.rn_hs + row], kp.inv_s2, kp.eps);
      if (MODE == TM_CROSS) {
        S = j.b.rho[bh + row];
        thr = __fmul_rn(kp.tau, j.b.base[bh + row]);
        if (S >= thr) cross = 0;
        snap_row = j.w.snap + (bh + row) * j.w.snap_stride;
        snap_row[0] = S;
      } else if (MODE == TM_PROJECT) {
        S = j.w.snap[(bh + row) * j.w.snap_stride + c0 / SNAP];
      } else if (MODE == TM_SUB) {
        slot = hd.e == 0 ? row : j.w.surv_list[bh + row];
      } else if (MODE == TM_NEWBASE) {
        self = j.w.slot_new[(int64_t)h * j.b.n_max + row];
      }
    }
    // column metadata source
    const float* cnorm = nullptr;
    const float* cbase = nullptr;
    if (MODE == TM_SCORE || MODE == TM_NEWBASE) cnorm = j.b.knorm + bh;
    if (MODE == TM_SCORE) cbase = j.b.base + bh;
    if (MODE == TM_CROSS || MODE == TM_PROJECT) cnorm = j.w.kperm_norm + (int64_t)h * j.b.n_max;
    if (MODE == TM_SUB) cnorm = j.w.kevict_norm + (int64_t)h * j.b.n_max;

    bool ok = true;
    for (int t = 0; t < ntiles; ++t) {
      const int b = t & 1;
      const int col0 = c0 + t * BN;
      const int nc = min(BN, c1 - col0);
      // stage this tile's column terms: cc = |k_j|^2 / sigma^2, and 1 / b_j for SCORE
      float* mc = meta + b * 2 * BN;
      {
        const int c = col0 + et;
        mc[et] = et < nc ? cnorm[c] * kp.inv_s2 : 0.f;
        if (MODE == TM_SCORE) mc[BN + et] = et < nc ? 1.0f / cbase[c] : 0.f;
      }
      // every epilogue warp takes this barrier on every tile, also after a failed wait,
      // so no warp is ever left waiting here
      named_bar(1, 128);
      if (ok) ok = __all_sync(0xffffffffu, mbar_wait(bar_accf + b, (t >> 1) & 1, abort_flag));
      if (!ok) continue;
      fence_after_sync();
      const uint32_t tbase = tmem + ((uint32_t)(q * 32) << 16) + b * BN;
#pragma unroll 1
      for (int c32 = 0; c32 < BN; c32 += 32) {
        if (c32 >= nc) break;
        float v[32];
        tmem_ld32(tbase + c32, v);
        tmem_wait_ld();
        if (!active) continue;
        const int lim = min(32, nc - c32);
#pragma unroll
        for (int jj = 0; jj < 32; ++jj) {
          if (jj < lim) {
            const float u = fmaxf(fmaf(v[jj], k2, cr + mc[c32 + jj]), kp.eps);
            const float r = rcp_approx(u);
            float w = r;
            if (kp.p >= 2) w = r * r;
            if (kp.p == 4) w = w * w;
            const int col = col0 + c32 + jj;
            if (MODE == TM_SCORE) {
              acc = fmaf(w, mc[BN + c32 + jj], acc);
            } else if (MODE == TM_CROSS) {
              S += w;
              if (cross == INT_MAX && S >= thr) cross = col + 1;
            } else if (MODE == TM_PROJECT) {
              S += w;
            } else if (MODE == TM_SUB) {
              acc += w;
            } else {
              if (col != self) S += w;
            }
          }
        }
      }
      if (MODE == TM_CROSS && active && nc == BN) snap_row[(col0 + BN) / SNAP] = S;
      fence_before_sync();
      __syncwarp();
      if (lane == 0) mbar_arrive(bar_acce + b);
    }
    if (!ok) {
      *abort_flag = 1;
      dev_fail(j.w.L, DEV_TIMEOUT, 300 + MODE);
    } else if (active) {
      if (MODE == TM_SCORE) {
        j.w.score[(int64_t)h * j.b.n_max + row] = acc / (float)hd.m_old;
      } else if (MODE == TM_CROSS) {
        j.w.cross[bh + row] = cross;
        const int bin = cross == INT_MAX ? L.rmax + 1 : cross;
        atomicAdd(&j.w.hist[(int64_t)h * j.w.hist_stride + bin], 1);
      } else if (MODE == TM_PROJECT) {
        j.w.rho_t[bh + row] = S;
      } else if (MODE == TM_SUB) {
        if (slot >= 0 && slot < hd.m_old) j.b.rho[bh + slot] = j.w.rho_t[bh + slot] - acc;
        else dev_fail(j.w.L, DEV_INCONSISTENT, 6003);
      } else {
        if (self >= 0 && self < hd.M) {
          j.b.rho[bh + self] = S;
          j.b.base[bh + self] = fmaxf(S, kp.delta);
        } else {
          dev_fail(j.w.L, DEV_INCONSISTENT, 6004);
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

// ---------------------------------------------------------------- host side
typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                  const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
  static EncodeTiledFn fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(p);
  });
  return fn;
}

}  // namespace

// bf16 [heads][rows][128] tensor, boxes of 64 columns x box_rows rows, 128-byte swizzle.
bool make_map_rows(CUtensorMap* m, const void* base, int64_t rows, int64_t heads, int box_rows) {
  EncodeTiledFn fn = encode_fn();
  if (!fn || rows < 1 || heads < 1) return false;
  cuuint64_t dims[3] = {128, (cuuint64_t)rows, (cuuint64_t)heads};
  cuuint64_t strides[2] = {256, (cuuint64_t)rows * 256};
  cuuint32_t box[3] = {64, (cuuint32_t)box_rows, 1};
  cuuint32_t es[3] = {1, 1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides, box, es,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

namespace {

template <int MODE>
cudaError_t launch_tc(const Bank& b, const Ws& w, const KParams& kp, const void* rk, int64_t rk_rows,
                      const float* rnorm, int64_t rn_hs, const void* ck, int64_t ck_rows, int max_rows,
                      cudaStream_t s, Timer* t, const char* name) {
  CUtensorMap ma, mb;
  if (!make_map_rows(&ma, rk, rk_rows, b.H, BM) || !make_map_rows(&mb, ck, ck_rows, b.H, BN))
    return cudaErrorInvalidValue;
  TcJob job{b, w, kp, rnorm, rn_hs};
  dim3 grid((max_rows + BM - 1) / BM, b.H);
  timer_begin(t, name, s);
  tc_pairs<MODE><<<grid, THREADS, SMEM_BYTES, s>>>(ma, mb, job);
  timer_end(t, s);
  return cudaGetLastError();
}

}  // namespace

bool tc_supported(int d, int bf16) { return d == 128 && bf16 && encode_fn() != nullptr; }

cudaError_t tc_attn_set_smem_limits();

cudaError_t tc_set_smem_limits() {
  cudaError_t e = cudaSuccess;
#define DKV_OPT(K) \
  if (e == cudaSuccess) e = cudaFuncSetAttribute(K, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)SMEM_BYTES)
  DKV_OPT(tc_pairs<TM_SCORE>);
  DKV_OPT(tc_pairs<TM_CROSS>);
  DKV_OPT(tc_pairs<TM_PROJECT>);
  DKV_OPT(tc_pairs<TM_SUB>);
  DKV_OPT(tc_pairs<TM_NEWBASE>);
#undef DKV_OPT
  if (e == cudaSuccess) e = tc_attn_set_smem_limits();
  return e;
}

cudaError_t launch_score_tc(const Bank& b, const Ws& w, const void* Kc, int N, const KParams& kp, cudaStream_t s,
                            Timer* t) {
  return launch_tc<TM_SCORE>(b, w, kp, Kc, N, w.cnorm, b.n_max, b.k, b.M_max, N, s, t, "score_tc");
}

cudaError_t launch_cross_tc(const Bank& b, const Ws& w, const KParams& kp, cudaStream_t s, Timer* t) {
  return launch_tc<TM_CROSS>(b, w, kp, b.k, b.M_max, b.knorm, b.M_max, w.kperm, b.n_max, b.M_max, s, t,
                             "cross_tc");
}

cudaError_t launch_project_tc(const Bank& b, const Ws& w, const KParams& kp, cudaStream_t s, Timer* t) {
  return launch_tc<TM_PROJECT>(b, w, kp, b.k, b.M_max, b.knorm, b.M_max, w.kperm, b.n_max, b.M_max, s, t,
                               "project_tc");
}

cudaError_t launch_subtract_tc(const Bank& b, const Ws& w, const KParams& kp, cudaStream_t s, Timer* t) {
  return launch_tc<TM_SUB>(b, w, kp, w.ksurv, b.M_max, w.ksurv_norm, b.M_max, w.kevict, b.n_max, b.M_max, s, t,
                           "subtract_tc");
}

cudaError_t launch_newbase_tc(const Bank& b, const Ws& w, const KParams& kp, cudaStream_t s, Timer* t) {
  return launch_tc<TM_NEWBASE>(b, w, kp, w.kperm, b.n_max, w.kperm_norm, b.n_max, b.k, b.M_max, b.n_max, s, t,
                               "newbase_tc");
}

}  // namespace dkv
