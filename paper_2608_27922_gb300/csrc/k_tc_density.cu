// Tensor-core (tcgen05) pair passes of the bank update, bf16 keys, d = 128.
//
// Every pass contracts a tile of 128 "row" keys against a run of "column" keys and
// folds the Soft-Riesz interaction (Eq. 2) into a per-row quantity in the
// epilogue, so no row-by-column matrix reaches global memory (App. C, "Decision
// granularity versus computational tiling"):
//   SCORE    rows = candidates, cols = bank:     s(x) = (1/m) sum_i w / b_i        (Eq. 6)
//   CROSS    rows = bank, cols = candidates in pi order: running rho~_i(r) (Eq. C.2)
//            and the first r with rho~_i(r) >= tau b_i (Eqs. 8-9); snapshots every
//            128 columns
//   PROJECT  rows = bank, cols = pi-ordered candidates [128 floor(r/128), r):
//            rho~_i(r), resumed from the snapshot with the same arithmetic
//   SUB      rows = survivors, cols = evicted:   rho_i = rho~_i - sum_R w       (Eq. C.4)
//   NEWBASE  rows = admitted, cols = final bank, self excluded by index:
//            rho_x = Phi(x), b_x = max(rho_x, delta)                     (Eq. 5 / C.4)
//
// Distances inside the MMA.  Each key carries 32 extension bf16 values (two forms
// of 16): row form [-g_hi, -g_mid, -g_lo, 1, 1, 1, 0..], column form
// [1, 1, 1, -h_hi, -h_mid, -h_lo, 0..] with g = |k|^2/2 + eps sigma^2/2 and
// h = |k|^2/2 split into three bf16 parts.  A ninth MMA k-step (K = 16) adds the
// product of the row form and the column form, so the fp32 accumulator holds
//   A = a.b - g_a - h_b = -(sigma^2/2) (eps + |a - b|^2 / sigma^2) = -(sigma^2/2) u,
// and w = u^-p = c |A|^-p with c = (sigma^2/2)^p.  Sums are kept in units of
// |A|^-p and scaled by c once per row.
//
// Epilogue arithmetic.  Two interactions share one reciprocal:
//   |A1|^-2 + |A2|^-2 = (A1^2 + A2^2) / (A1 A2)^2,
// and the 16 pair terms of a 32-column chunk are accumulated in a fixed order: two
// independent chains of four packed fp32x2 accumulations, added at the end, so a
// chunk's dependence chain is short.  The crossing pass tests each chunk total
// against the row's threshold and rescans a chunk term by term only when the
// threshold falls inside it (at most once per row).
//
// CTA (320 threads, 2 per SM): warp 0 TMA producer, warp 1 MMA issuer, warps 2-9
// epilogue.  Epilogue warps w and w+4 share TMEM lanes 32 (w % 4) .. +31 (one row
// per lane) and split each 128-column tile into halves of 64 columns; the crossing
// and projection passes exchange half totals through shared memory every tile.
// Persistent forms (one CTA per SM, or two, taking units in turn): the crossing pass
// over keys with two row tiles per unit (tc_cross_dual), the score pass over many
// candidate row tiles with 256-column bank tiles (tc_score_wide), and the projection,
// survivor and new-baseline passes over many row tiles (tc_pairs_loop); the [K; V]
// descriptor keeps the one-row-tile form.
#include "dkv_internal.h"
#include "tc_ptx.cuh"

#include <algorithm>
#include <climits>
#include <mutex>

namespace dkv {

namespace {

using namespace tc;

enum TMode { TM_SCORE = 0, TM_CROSS = 1, TM_PROJECT = 2, TM_SUB = 3, TM_NEWBASE = 4 };

constexpr int BM = 128;                     // rows per CTA (TMEM lanes)
constexpr int BN = 128;                     // columns per tile
constexpr int HALF_BYTES = BM * 64 * 2;    // one 64-column 128-byte-swizzle panel (16 KiB)
constexpr int EXT_BYTES = BM * 16 * 2;      // 128 rows x 16 bf16 (32-byte swizzle)
constexpr int STAGES = 2;
constexpr int EPI_WARPS = 8;
constexpr int THREADS = 64 + 32 * EPI_WARPS;
constexpr uint32_t TMEM_COLS = 256;         // two 128-column accumulators
// score weights of tiles t .. t+4: buffer t % 5 is refilled for tile t + 5 once the MMA
// of tile t + 3 has completed, which needs every epilogue warp's release of tile t + 1,
// given only after that warp finished tile t (the release can precede a tile's arithmetic)
constexpr int META_BUFS = 5;

// Shared-memory layout.  A tile row is the state's descriptor: its key (two 64-column
// panels) or, with the [K; V] descriptor (App. E), its key and value (four panels); one
// CTA per SM then (209 KiB), two otherwise (2 x 110 KiB).
template <bool KV>
struct Lay {
  static constexpr int NP = KV ? 4 : 2;                        // 64-column panels per row
  static constexpr int TILE = NP * HALF_BYTES;
  static constexpr int A = 0;
  static constexpr int AX = TILE;
  static constexpr int B = AX + EXT_BYTES;                     // [STAGES] tiles
  static constexpr int BX = B + STAGES * TILE;                 // [STAGES] extension tiles
  static constexpr int META = BX + STAGES * EXT_BYTES;         // float [META_BUFS][BN]
  static constexpr int XCH = META + META_BUFS * BN * 4;        // float [2][2][BM]
  static constexpr int FLAG = XCH + 2 * 2 * BM * 4;            // int: last-arrival flag of split tiles
  static constexpr int BAR = FLAG + 16;
  static constexpr size_t SMEM = BAR + 128;                    // base 1024-aligned (checked)
  static constexpr uint32_t LOAD = TILE + EXT_BYTES;
  static_assert(B % 1024 == 0 && TILE % 1024 == 0, "128-byte-swizzled panels need 1024-byte alignment");
  static_assert(SMEM <= 227 * 1024, "shared memory per CTA");
};

struct TcJob {
  Bank b;
  Ws w;
  KParams kp;
  int lin;   // 1: row tiles are the budget-sized 128-row tiles of all heads (w.tile_head)
  int tpn;   // row tiles per head otherwise (persistent kernel: unit u = head u / tpn, tile u % tpn)
};

// Head and row tile of work unit u of the persistent kernel.
__device__ __forceinline__ void unit_of(const TcJob& j, int u, int& h, int& rtile) {
  if (j.lin) {
    h = j.w.tile_head[u];
    rtile = u - j.w.tile_first[h];
  } else {
    h = u / j.tpn;
    rtile = u - h * j.tpn;
  }
}

// (sigma^2 / 2)^P: the scale between |A|^-P and w (Eq. 2 through the MMA).
template <int P>
__device__ __forceinline__ float pow_c(const KParams& kp) {
  const float hs2 = 0.5f / kp.inv_s2;
  float c = hs2;
  if (P >= 2) c = hs2 * hs2;
  if (P == 4) c = c * c;
  return c;
}

__device__ __forceinline__ void job_range(int MODE, const DevHead& hd, const DevLayer& L, int& nrows, int& c0,
                                          int& c1) {
  nrows = 0; c0 = 0; c1 = 0;
  if (MODE == TM_SCORE) { nrows = hd.empty ? 0 : L.N; c1 = hd.m_old; }
  if (MODE == TM_CROSS) { nrows = hd.empty ? 0 : hd.m_old; c1 = L.rmax; }
  if (MODE == TM_PROJECT) { nrows = hd.empty ? 0 : hd.m_old; c0 = (hd.r / SNAP) * SNAP; c1 = hd.r; }
  if (MODE == TM_SUB) { nrows = hd.empty ? 0 : hd.m_old - hd.e; c1 = hd.e; }
  if (MODE == TM_NEWBASE) { nrows = hd.r; c1 = hd.m_new; }
}

// |a|^-P for a < 0 (one reciprocal).
template <int P>
__device__ __forceinline__ float term1(float a) {
  const float r = rcp_approx(a);
  if (P == 1) return -r;
  const float r2 = r * r;
  return P == 2 ? r2 : r2 * r2;
}

// Two interactions X, Y < 0 share one reciprocal R = 1 / (X Y):
//   |X|^-2 + |Y|^-2 = (X^2 + Y^2) R^2,   wX |X|^-2 + wY |Y|^-2 = (wX Y^2 + wY X^2) R^2,
// in packed fp32x2 arithmetic (lane l of X and Y holds one pair; each lane rounds
// exactly like the scalar expression), the last multiply fused into the accumulation:
// acc += |X|^-P + |Y|^-P per lane.  For P = 1 the accumulator collects
// (X + Y) / (X Y) = -(|X|^-1 + |Y|^-1); the caller negates the chunk total.
template <int P>
__device__ __forceinline__ float2 acc2x2(float2 X, float2 Y, float2 acc) {
  const float2 Pm = __fmul2_rn(X, Y);
  const float2 R = make_float2(rcp_approx(Pm.x), rcp_approx(Pm.y));
  if (P == 1) return __ffma2_rn(R, __fadd2_rn(X, Y), acc);
  const float2 R2 = __fmul2_rn(R, R);
  if (P == 2) return __ffma2_rn(R2, __ffma2_rn(X, X, __fmul2_rn(Y, Y)), acc);
  const float2 X2 = __fmul2_rn(X, X), Y2 = __fmul2_rn(Y, Y);
  return __ffma2_rn(__fmul2_rn(R2, R2), __ffma2_rn(X2, X2, __fmul2_rn(Y2, Y2)), acc);
}

// acc += wX |X|^-P + wY |Y|^-P per lane (same conventions).
template <int P>
__device__ __forceinline__ float2 acc2wx2(float2 X, float2 Y, float2 WX, float2 WY, float2 acc) {
  const float2 Pm = __fmul2_rn(X, Y);
  const float2 R = make_float2(rcp_approx(Pm.x), rcp_approx(Pm.y));
  if (P == 1) return __ffma2_rn(R, __ffma2_rn(WX, Y, __fmul2_rn(WY, X)), acc);
  const float2 R2 = __fmul2_rn(R, R);
  if (P == 2) return __ffma2_rn(R2, __ffma2_rn(WX, __fmul2_rn(Y, Y), __fmul2_rn(WY, __fmul2_rn(X, X))), acc);
  const float2 X2 = __fmul2_rn(X, X), Y2 = __fmul2_rn(Y, Y);
  return __ffma2_rn(__fmul2_rn(R2, R2), __ffma2_rn(WX, __fmul2_rn(Y2, Y2), __fmul2_rn(WY, __fmul2_rn(X2, X2))),
                    acc);
}

// Sum of |v_j|^-P over a full 32-column chunk: column j shares a reciprocal with
// column j + 16; two packed accumulators (even and odd pairs), added at the end.
template <int P>
__device__ __forceinline__ float chunk_sum(const float (&v)[32]) {
  float2 a0 = make_float2(0.f, 0.f), a1 = make_float2(0.f, 0.f);
#pragma unroll
  for (int k = 0; k < 8; k += 2) {
    a0 = acc2x2<P>(make_float2(v[2 * k], v[2 * k + 1]), make_float2(v[2 * k + 16], v[2 * k + 17]), a0);
    a1 = acc2x2<P>(make_float2(v[2 * k + 2], v[2 * k + 3]), make_float2(v[2 * k + 18], v[2 * k + 19]), a1);
  }
  const float2 a = __fadd2_rn(a0, a1);
  return P == 1 ? -(a.x + a.y) : a.x + a.y;
}

// Score pass, one warp's 64-column half of a tile in the 16x256b layout (va: lanes
// 0..15 of the warp's quarter, vb: lanes 16..31): this thread holds rows i/4, i/4 + 8,
// i/4 + 16, i/4 + 24 at columns 8k + 2 (i % 4) + {0, 1}, k = 0..7, so it needs 16
// weights for 4 rows.  acc[j] += sum of wb_c |v|^-P over row j's columns, in the
// accumulation convention of acc2wx2 (negated for P = 1); columns from lim on are left
// out (term by term in a partial tile).
template <int P>
__device__ __forceinline__ void score_rows4(const float (&va)[32], const float (&vb)[32], const float* wb, int lim,
                                            int c2, float2 (&acc)[4]) {
  if (lim >= 64) {
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      const float2 w0 = *reinterpret_cast<const float2*>(wb + 8 * k + c2);
      const float2 w1 = *reinterpret_cast<const float2*>(wb + 8 * (k + 4) + c2);
      acc[0] = acc2wx2<P>(make_float2(va[4 * k], va[4 * k + 1]), make_float2(va[4 * k + 16], va[4 * k + 17]), w0, w1,
                          acc[0]);
      acc[1] = acc2wx2<P>(make_float2(va[4 * k + 2], va[4 * k + 3]), make_float2(va[4 * k + 18], va[4 * k + 19]), w0,
                          w1, acc[1]);
      acc[2] = acc2wx2<P>(make_float2(vb[4 * k], vb[4 * k + 1]), make_float2(vb[4 * k + 16], vb[4 * k + 17]), w0, w1,
                          acc[2]);
      acc[3] = acc2wx2<P>(make_float2(vb[4 * k + 2], vb[4 * k + 3]), make_float2(vb[4 * k + 18], vb[4 * k + 19]), w0,
                          w1, acc[3]);
    }
    return;
  }
  const float sg = P == 1 ? -1.f : 1.f;
#pragma unroll
  for (int k = 0; k < 8; ++k)
#pragma unroll
    for (int e = 0; e < 2; ++e) {
      const int c = 8 * k + c2 + e;
      if (c < lim) {
        const float w = sg * wb[c];
        acc[0].x = fmaf(term1<P>(va[4 * k + e]), w, acc[0].x);
        acc[1].x = fmaf(term1<P>(va[4 * k + 2 + e]), w, acc[1].x);
        acc[2].x = fmaf(term1<P>(vb[4 * k + e]), w, acc[2].x);
        acc[3].x = fmaf(term1<P>(vb[4 * k + 2 + e]), w, acc[3].x);
      }
    }
}

// Same over the first `lim` columns (lim < 32), term by term.
template <int P>
__device__ __forceinline__ float chunk_sum_partial(const float (&v)[32], int lim) {
  float s = 0.f;
#pragma unroll
  for (int j = 0; j < 32; ++j)
    if (j < lim) s += term1<P>(v[j]);
  return s;
}

// Sum over `lim` columns skipping column `skip` (-1: none), term by term.
template <int P>
__device__ __forceinline__ float chunk_sum_skip(const float (&v)[32], int lim, int skip) {
  float s = 0.f;
#pragma unroll
  for (int j = 0; j < 32; ++j)
    if (j < lim && j != skip) s += term1<P>(v[j]);
  return s;
}

// TMEM of the pair passes: warp 1 allocates TMEM_COLS columns (and gives up the CTA's
// allocation permit) into the holder word of the barrier area; every thread returns the
// address.  Called by all threads of the CTA together, as is cta_tmem_free.
__device__ __forceinline__ uint32_t cta_tmem_alloc(uint8_t* bar_area) {
  uint32_t* holder = reinterpret_cast<uint32_t*>(reinterpret_cast<uint64_t*>(bar_area) + 9);
  if ((threadIdx.x >> 5) == 1) tmem_alloc(holder, TMEM_COLS);
  fence_before_sync();
  __syncthreads();
  fence_after_sync();
  return *holder;
}

__device__ __forceinline__ void cta_tmem_free(uint32_t tmem) {
  fence_before_sync();
  __syncthreads();
  if ((threadIdx.x >> 5) == 1) {
    fence_after_sync();
    tmem_dealloc(tmem, TMEM_COLS);
  }
}

// A row of a pass that has no column at all (projection at a prefix length that is a
// multiple of the snapshot spacing, survivor maintenance without evictions): the row keeps
// its running sum and is finished exactly as the epilogue finishes it after no tile; no
// MMA, TMEM or barrier.
template <int MODE, int P>
__device__ __forceinline__ void trivial_row(const TcJob& j, const DevHead& hd, int h, int row, int c0) {
  const int64_t bh = (int64_t)h * j.b.M_max;
  const float c = pow_c<P>(j.kp);
  if (MODE == TM_PROJECT) {
    // the snapshot at column 0 is the empty sum, 0 (written by the crossing pass): rows of
    // a prefix shorter than a snapshot spacing skip its strided load
    const float S = c0 == 0 ? 0.f : j.w.snap[(bh + row) * j.w.snap_stride + c0 / SNAP];
    j.w.rho_t[bh + row] = fmaf(c, S, j.b.rho[bh + row]);
  } else if (MODE == TM_SUB) {
    const int slot = hd.e == 0 ? row : j.w.surv_list[bh + row];
    if (slot >= 0 && slot < hd.m_old) {
      const float rho = fmaf(-c, 0.f, j.w.rho_t[bh + slot]);
      j.b.rho[bh + slot] = rho;
      if (j.kp.refresh) {
        const float bnew = fmaxf(rho, j.kp.delta);
        j.b.base[bh + slot] = bnew;
        j.w.invb[(int64_t)h * j.w.invb_stride + slot] = __frcp_rn(bnew);
      }
    } else {
      dev_fail(j.w.L, DEV_INCONSISTENT, 6003);
    }
  }
}

// One row tile (rows [128 rtile, +128) of head h) against its column tiles, columns split
// over nz CTAs of which this is number zi, in the CTA's TMEM columns [tmem, tmem + 256)
// (allocated once per CTA by the caller: a CTA may allocate only until it relinquishes
// its allocation permit).  Every thread of the CTA calls it together; it leaves the
// shared-memory barriers invalidated.  Returns false if a bounded wait gave up.
template <int MODE, int P, bool KV>
__device__ __forceinline__ bool pairs_unit(const CUtensorMap& tmA, const CUtensorMap& tmAx, const CUtensorMap& tmB,
                                           const CUtensorMap& tmBx, const CUtensorMap& tmAv, const CUtensorMap& tmBv,
                                           const TcJob& j, uint8_t* smem, uint32_t tmem, int h, int rtile, int zi,
                                           int nz) {
  using LY = Lay<KV>;
  float* meta = reinterpret_cast<float*>(smem + LY::META);
  float* xch = reinterpret_cast<float*>(smem + LY::XCH);
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + LY::BAR);
  uint64_t* bar_a = bars + 0;
  // ready[b]: column tile t (b = t & 1) has landed AND the epilogue has released
  // accumulator b (tile t - 2): the MMA issuer's only wait per tile
  uint64_t* bar_rdy = bars + 1;     // [2]
  uint64_t* bar_empty = bars + 3;   // [STAGES] MMA of the stage's tile complete
  uint64_t* bar_accf = bars + 5;    // [2] accumulator b complete
  uint32_t* tmem_holder = reinterpret_cast<uint32_t*>(bars + 9);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_holder + 1);
  uint64_t* bar_meta = bars + 10;   // [META_BUFS] SCORE: 1 / b of the columns of tile t (t % 4)

  const DevHead hd = j.w.hd[h];
  const DevLayer L = *layer_of(j.w, h);
  int nrows, c0, c1;
  job_range(MODE, hd, L, nrows, c0, c1);
  const int row0 = rtile * BM;
  // column tiles of this CTA: the row passes with plain row sums may split the column
  // range over nz CTAs (their partial sums are combined below)
  const int ntot = c1 > c0 ? (c1 - c0 + BN - 1) / BN : 0;
  const int per = (ntot + nz - 1) / nz;
  const int tbeg = min(ntot, zi * per);
  const int ntiles = min(ntot, tbeg + per) - tbeg;
  c0 += tbeg * BN;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    mbar_init(bar_a, 1);
    for (int s = 0; s < STAGES; ++s) mbar_init(bar_empty + s, 1);
    for (int b = 0; b < 2; ++b) {
      mbar_init(bar_accf + b, 1);
      mbar_init(bar_rdy + b, EPI_WARPS + 1);   // the epilogue warps + the producer (with bytes)
    }
    for (int q = 0; q < META_BUFS; ++q) mbar_init(bar_meta + q, 1);
    *abort_flag = 0;
    fence_barrier_init();
  }
  fence_before_sync();
  __syncthreads();
  fence_after_sync();

  if (warp == 0) {
    if (lane == 0 && ntiles > 0) {
      // ---------------- TMA producer: row tile (+ row-form extension) once, column tiles
      prefetch_map(&tmA); prefetch_map(&tmAx); prefetch_map(&tmB); prefetch_map(&tmBx);
      if (KV) { prefetch_map(&tmAv); prefetch_map(&tmBv); }
      mbar_arrive_expect_tx(bar_a, LY::LOAD);
#pragma unroll
      for (int pn = 0; pn < LY::NP; ++pn)   // key panels, then value panels ([K; V])
        tma_load_3d(smem + LY::A + pn * HALF_BYTES, pn < 2 ? &tmA : &tmAv, bar_a, (pn & 1) * 64, row0, h);
      tma_load_3d(smem + LY::AX, &tmAx, bar_a, 0, row0, h);
      int issued = 0;
      for (int t = 0; t < ntiles; ++t) {
        const int s = t % STAGES;   // == t & 1, the accumulator of tile t
        // MMA(t - 2) complete: stage s is free, and (it waited for ready) the epilogue of
        // tile t - 4 has finished with meta buffer t % 4
        if (!mbar_wait(bar_empty + s, ((t / STAGES) & 1) ^ 1, abort_flag)) break;
        mbar_arrive_expect_tx(bar_rdy + s, LY::LOAD);
        const int col = c0 + t * BN;
        uint8_t* dst = smem + LY::B + s * LY::TILE;
#pragma unroll
        for (int pn = 0; pn < LY::NP; ++pn)
          tma_load_3d(dst + pn * HALF_BYTES, pn < 2 ? &tmB : &tmBv, bar_rdy + s, (pn & 1) * 64, col, h);
        tma_load_3d(smem + LY::BX + s * EXT_BYTES, &tmBx, bar_rdy + s, 16, col, h);
        if (MODE == TM_SCORE) {
          // 1 / b_j of the tile's columns (a whole 128-float row; values past the last
          // column are not used)
          const int q = t % META_BUFS;
          mbar_arrive_expect_tx(bar_meta + q, BN * 4);
          bulk_load(meta + q * BN, j.w.invb + (int64_t)h * j.w.invb_stride + col, BN * 4, bar_meta + q);
        }
        issued = t + 1;
      }
      if (issued < ntiles) {
        *abort_flag = 1;
        dev_fail(j.w.L, DEV_TIMEOUT, 100 + MODE);
      }
      // never leave with copies in flight: wait (bounded) for the last loads issued.  A
      // ready phase also needs the epilogue's release, which an aborted CTA may never
      // give; then wait a fixed 50 us, far longer than any copy takes to land.
      volatile int no_abort = 0;
      mbar_wait(bar_a, 0, &no_abort);
      bool drained = true;
      for (int t = issued > STAGES ? issued - STAGES : 0; t < issued; ++t)
        drained = drained && mbar_wait(bar_rdy + (t % STAGES), (t / STAGES) & 1, abort_flag);
      if (MODE == TM_SCORE)
        for (int t = issued > META_BUFS ? issued - META_BUFS : 0; t < issued; ++t)
          mbar_wait(bar_meta + (t % META_BUFS), (t / META_BUFS) & 1, &no_abort);
      if (!drained) {
        const uint64_t t0 = globaltimer_ns();
        while (globaltimer_ns() - t0 < 50000ull) {
        }
      }
    }
  } else if (warp == 1) {
    if (lane == 0 && ntiles > 0) {
      // ---------------- MMA issuer: 8 k-steps per key (16 per [key; value]) + 1 of the extension
      constexpr uint32_t idesc = idesc_bf16(BM, BN);
      bool ok = mbar_wait(bar_a, 0, abort_flag);
      // every operand's descriptor once; the k-steps' by one add each (desc_add)
      const uint64_t ad0 = desc_sw128(smem_u32(smem + LY::A));
      const uint64_t axd = desc_sw32(smem_u32(smem + LY::AX));
      const uint64_t bd0 = desc_sw128(smem_u32(smem + LY::B));
      const uint64_t bxd0 = desc_sw32(smem_u32(smem + LY::BX));
      int done = 0;
      for (int t = 0; ok && t < ntiles; ++t) {
        const int s = t % STAGES;
        const int b = t & 1;
        // one wait per tile: every other wait in this thread stalls the tensor pipe
        if (!(ok = mbar_wait(bar_rdy + b, (t >> 1) & 1, abort_flag))) break;
        fence_after_sync();
        const uint64_t bd = desc_add(bd0, s * LY::TILE);
#pragma unroll
        for (int kk = 0; kk < 4 * LY::NP; ++kk) {
          const uint32_t koff = (kk >> 2) * HALF_BYTES + (kk & 3) * 32;
          mma_bf16(tmem + b * BN, desc_add(ad0, koff), desc_add(bd, koff), idesc, kk > 0);
        }
        mma_bf16(tmem + b * BN, axd, desc_add(bxd0, s * EXT_BYTES), idesc, 1u);
        mma_commit(bar_empty + s);
        mma_commit(bar_accf + b);
        done = t + 1;
      }
      if (!ok) {
        *abort_flag = 1;
        dev_fail(j.w.L, DEV_TIMEOUT, 200 + MODE);
      }
      // all issued MMAs must be complete before TMEM is freed, and no copy may be in flight
      if (done > 0) {
        volatile int no_abort = 0;
        mbar_wait(bar_accf + ((done - 1) & 1), ((done - 1) >> 1) & 1, &no_abort);
      }
    }
  } else {
    // ---------------- epilogue: thread = row (TMEM lane); two warps per row quarter
    const int ew = warp - 2;                      // 0..7
    const int half = ew >> 2;                     // columns [64 half, 64 half + 64) of each tile
    const int q = warp & 3;                       // TMEM lane quarter
    const int r_local = q * 32 + lane;
    const int row = row0 + r_local;
    const bool active = row < nrows;
    const int et = threadIdx.x - 64;              // 0..255
    const int64_t bh = (int64_t)h * j.b.M_max;
    const KParams kp = j.kp;
    const float c = pow_c<P>(kp);                 // (sigma^2 / 2)^p
    const uint32_t lane_base = tmem + ((uint32_t)(q * 32) << 16);
    // per-row state (sums in units of |A|^-p)
    float S = 0.f, acc = 0.f, thr = 0.f;
    int cross = INT_MAX, self = -1;
    float* snap_row = nullptr;
    if (active) {
      if (MODE == TM_CROSS) {
        const float rho = j.b.rho[bh + row];
        thr = (__fmul_rn(kp.tau, j.b.base[bh + row]) - rho) / c;
        if (thr <= 0.f) cross = 0;
        snap_row = j.w.snap + (bh + row) * j.w.snap_stride;
      } else if (MODE == TM_PROJECT) {
        S = j.w.snap[(bh + row) * j.w.snap_stride + c0 / SNAP];
      } else if (MODE == TM_NEWBASE) {
        self = j.w.slot_new[(int64_t)h * j.b.n_max + row];
      }
    }
    if (MODE == TM_CROSS && active && half == 0) snap_row[0] = 0.f;
    // both accumulators start free: this warp's release for tiles 0 and 1
    if (lane == 0) {
      mbar_arrive(bar_rdy + 0);
      mbar_arrive(bar_rdy + 1);
    }

    float2 sacc[4];   // score pass: rows lane/4 + 8 j of the quarter (16x256b layout)
#pragma unroll
    for (int jj = 0; jj < 4; ++jj) sacc[jj] = make_float2(0.f, 0.f);
    bool ok = true;
    for (int t = 0; t < ntiles; ++t) {
      const int b = t & 1;
      const int col0 = c0 + t * BN;
      const int nc = min(BN, c1 - col0);
      if (ok) ok = __all_sync(0xffffffffu, mbar_wait(bar_accf + b, (t >> 1) & 1, abort_flag));
      if (MODE == TM_SCORE && ok)
        ok = __all_sync(0xffffffffu,
                        mbar_wait(bar_meta + t % META_BUFS, (t / META_BUFS) & 1, abort_flag));
      float tot[2] = {0.f, 0.f};
      constexpr bool kEarlyRelease = MODE == TM_SCORE || MODE == TM_SUB || MODE == TM_NEWBASE;
      if (ok && MODE == TM_SCORE) {
        fence_after_sync();
        const int cs = half * 64;
        if (cs < nc) {   // warp-uniform
          float va[32], vb[32];
          tmem_ld16x256b_x8(lane_base + b * BN + cs, va);
          tmem_ld16x256b_x8(lane_base + (16u << 16) + b * BN + cs, vb);
          tmem_wait_ld();
          fence_before_sync();
          __syncwarp();
          if (lane == 0) mbar_arrive(bar_rdy + b);   // accumulator b free for tile t + 2
          score_rows4<P>(va, vb, meta + (t % META_BUFS) * BN + cs, nc - cs, 2 * (lane & 3), sacc);
        }
      } else if (ok) {
        fence_after_sync();
#pragma unroll
        for (int ch = 0; ch < 2; ++ch) {
          const int cs = half * 64 + ch * 32;     // first column of the chunk within the tile
          if (cs >= nc) continue;                 // warp-uniform
          float v[32];
          tmem_ld32(lane_base + b * BN + cs, v);
          tmem_wait_ld();
          // row-sum passes: after the warp's last TMEM load of the tile the accumulator is
          // released before that chunk's arithmetic (the values are in registers; loading
          // both chunks before one wait measured slower: survivor pass 0.068 -> 0.077 ms at
          // config 1)
          if (kEarlyRelease && (ch == 1 || cs + 32 >= nc)) {
            fence_before_sync();
            __syncwarp();
            if (lane == 0) mbar_arrive(bar_rdy + b);   // accumulator b free for tile t + 2
          }
          const int lim = min(32, nc - cs);
          if (MODE == TM_NEWBASE) {   // (the score pass takes the 16x256b branch above)
            const int sk = self - (col0 + cs);
            if (lim == 32 && (sk < 0 || sk >= 32)) tot[ch] = chunk_sum<P>(v);
            else tot[ch] = chunk_sum_skip<P>(v, lim, sk);
          } else {
            tot[ch] = lim == 32 ? chunk_sum<P>(v) : chunk_sum_partial<P>(v, lim);
          }
        }
      }
      if (MODE == TM_CROSS || MODE == TM_PROJECT) {
        // exchange the half totals of this row, so both warps carry the same running sum
        const float mine = tot[0] + tot[1];
        xch[(b * 2 + half) * BM + r_local] = mine;
        named_bar(1 + q, 64);
        const float other = xch[(b * 2 + (half ^ 1)) * BM + r_local];
        const float T0 = half == 0 ? mine : other;
        const float T1 = half == 0 ? other : mine;
        if (MODE == TM_CROSS && ok) {
          const float base0 = half == 0 ? S : S + T0;
          int hit = -1;
          float run = base0;
          if (active && cross == INT_MAX) {
            if (base0 + tot[0] >= thr) hit = 0;
            else if ((base0 + tot[0]) + tot[1] >= thr) { hit = 1; run = base0 + tot[0]; }
          }
          // exact position inside the chunk, term by term (at most once per row); the
          // TMEM load is warp-collective, so the whole warp takes part for each chunk hit
#pragma unroll
          for (int hc = 0; hc < 2; ++hc) {
            const int cs = half * 64 + hc * 32;
            if (cs < nc && __any_sync(0xffffffffu, hit == hc)) {
              float v[32];
              tmem_ld32(lane_base + b * BN + cs, v);
              tmem_wait_ld();
              if (hit == hc) {
                const int lim = min(32, nc - cs);
                // the 32 terms are independent: all of them first (in place), then the
                // running sum
#pragma unroll
                for (int jj = 0; jj < 32; ++jj) v[jj] = term1<P>(v[jj]);
                int pos = lim;
#pragma unroll
                for (int jj = 0; jj < 32; ++jj) {
                  if (jj < lim && pos == lim) {
                    run += v[jj];
                    if (run >= thr) pos = jj + 1;
                  }
                }
                cross = col0 + cs + pos;
              }
            }
          }
        }
        S = (S + T0) + T1;
        if (MODE == TM_CROSS && ok && active && half == 0 && nc == BN) snap_row[(col0 + BN) / SNAP] = S;
      } else {
        acc += tot[0] + tot[1];
      }
      // a warp whose half lies past the tile's last column loaded nothing: release here too
      if (ok && (!kEarlyRelease || half * 64 >= nc)) {
        fence_before_sync();
        __syncwarp();
        if (lane == 0) mbar_arrive(bar_rdy + b);   // accumulator b free for tile t + 2
      }
    }
    if (!ok) {
      *abort_flag = 1;
      if (lane == 0) dev_fail(j.w.L, DEV_TIMEOUT, 300 + MODE);
    }
    bool finalize = true;
    if (MODE == TM_SCORE || MODE == TM_SUB || MODE == TM_NEWBASE) {
      // combine the two column halves of each row (no per-tile exchange in these passes)
      if (MODE == TM_SCORE) {
        // the four threads of a row quad hold a quarter of the half's columns each
#pragma unroll
        for (int jj = 0; jj < 4; ++jj) {
          float x = sacc[jj].x + sacc[jj].y;
          x += __shfl_xor_sync(0xffffffffu, x, 1);
          x += __shfl_xor_sync(0xffffffffu, x, 2);
          if ((lane & 3) == 0) xch[half * BM + q * 32 + (lane >> 2) + 8 * jj] = P == 1 ? -x : x;
        }
      } else {
        xch[half * BM + r_local] = acc;
      }
      named_bar(1 + q, 64);
      acc = xch[r_local] + xch[BM + r_local];
      if (nz > 1) {
        // column-split row tile: publish this CTA's partial; the last CTA of the tile to
        // arrive adds the partials in split order and finishes the rows
        float* part = j.w.part + (int64_t)h * j.w.part_stride;
        const int64_t zstride = (int64_t)j.b.H * j.w.part_stride;
        if (half == 0 && active) part[zi * zstride + row] = acc;
        __threadfence();
        named_bar(6, 32 * EPI_WARPS);
        int* flag = reinterpret_cast<int*>(smem + LY::FLAG);
        if (et == 0) {
          int32_t* cnt = j.w.cnt + (int64_t)h * j.w.cnt_stride + rtile;
          const int prev = atomicAdd(cnt, 1);
          const int last = prev == nz - 1;
          if (last) atomicExch(cnt, 0);
          *flag = last;
        }
        named_bar(6, 32 * EPI_WARPS);
        finalize = *flag != 0;
        if (finalize) {
          __threadfence();
          if (half == 0 && active) {
            float sum = 0.f;
            for (int z = 0; z < nz; ++z) sum += __ldcg(part + z * zstride + row);
            acc = sum;
          }
        }
      }
    }
    if (MODE == TM_CROSS) {
      // each half saw only its own columns: the row's first crossing is the earlier one.
      // The exchange slots of parity (ntiles & 1) were last read before the final tile's
      // barrier, so they are free.
      int* xi = reinterpret_cast<int*>(xch) + (ntiles & 1) * 2 * BM;
      xi[half * BM + r_local] = cross;
      named_bar(1 + q, 64);
      cross = min(xi[r_local], xi[BM + r_local]);
    }
    if (ok && finalize && active && half == 0) {
      if (MODE == TM_SCORE) {
        j.w.score[(int64_t)h * j.b.n_max + row] = (acc * c) / (float)hd.m_old;
      } else if (MODE == TM_CROSS) {
        j.w.cross[bh + row] = cross;
        const int bin = cross == INT_MAX ? L.rmax + 1 : cross;
        atomicAdd(&j.w.hist[(int64_t)h * j.w.hist_stride + bin], 1);
      } else if (MODE == TM_PROJECT) {
        j.w.rho_t[bh + row] = fmaf(c, S, j.b.rho[bh + row]);
      } else if (MODE == TM_SUB) {
        const int slot = hd.e == 0 ? row : j.w.surv_list[bh + row];
        if (slot >= 0 && slot < hd.m_old) {
          const float rho = fmaf(-c, acc, j.w.rho_t[bh + slot]);
          j.b.rho[bh + slot] = rho;
          if (kp.refresh) {   // refreshed-baseline policy: b follows the current density
            const float bnew = fmaxf(rho, kp.delta);
            j.b.base[bh + slot] = bnew;
            j.w.invb[(int64_t)h * j.w.invb_stride + slot] = __frcp_rn(bnew);
          }
        } else {
          dev_fail(j.w.L, DEV_INCONSISTENT, 6003);
        }
      } else {
        if (self >= 0 && self < hd.M) {
          const float rho = c * acc;
          j.b.rho[bh + self] = rho;
          const float bnew = fmaxf(rho, kp.delta);
          j.b.base[bh + self] = bnew;
          j.w.invb[(int64_t)h * j.w.invb_stride + self] = __frcp_rn(bnew);
        } else {
          dev_fail(j.w.L, DEV_INCONSISTENT, 6004);
        }
      }
    }
  }
  fence_before_sync();
  __syncthreads();
  const bool unit_ok = *abort_flag == 0;
  if (threadIdx.x == 0) {   // the barriers may be initialised again for the next unit
    mbar_inval(bar_a);
    for (int b = 0; b < 2; ++b) {
      mbar_inval(bar_rdy + b);
      mbar_inval(bar_accf + b);
    }
    for (int s = 0; s < STAGES; ++s) mbar_inval(bar_empty + s);
    for (int q = 0; q < META_BUFS; ++q) mbar_inval(bar_meta + q);
  }
  __syncthreads();
  return unit_ok;
}

template <int MODE, int P, bool KV>
__global__ void __launch_bounds__(THREADS, KV ? 1 : 2)
    tc_pairs(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmAx,
             const __grid_constant__ CUtensorMap tmB, const __grid_constant__ CUtensorMap tmBx,
             const __grid_constant__ CUtensorMap tmAv, const __grid_constant__ CUtensorMap tmBv, TcJob j) {
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  if ((smem_u32(smem_raw) & 1023u) != 0u) {   // 128-byte-swizzled tiles need 1024-byte alignment
    if (threadIdx.x == 0) dev_fail(j.w.L, DEV_INCONSISTENT, 9900);
    return;
  }
  // row tile: (blockIdx.x, head blockIdx.y), or the blockIdx.x-th budget-sized row tile
  // of all heads (the passes whose rows are bank states: no CTA for rows past a head's budget)
  const int h = j.lin ? j.w.tile_head[blockIdx.x] : (int)blockIdx.y;
  const int rtile = j.lin ? (int)blockIdx.x - j.w.tile_first[h] : (int)blockIdx.x;
  const DevHead hd = j.w.hd[h];
  int nrows, c0, c1;
  job_range(MODE, hd, *layer_of(j.w, h), nrows, c0, c1);
  const int row0 = rtile * BM;
  if (row0 >= nrows) return;                      // uniform: before any barrier or TMEM use
  if (c1 <= c0 && (MODE == TM_PROJECT || MODE == TM_SUB)) {
    const int row = row0 + (int)threadIdx.x;
    if (threadIdx.x < BM && row < nrows) trivial_row<MODE, P>(j, hd, h, row, c0);
    return;
  }
  const uint32_t tmem = cta_tmem_alloc(smem_raw + Lay<KV>::BAR);
  pairs_unit<MODE, P, KV>(tmA, tmAx, tmB, tmBx, tmAv, tmBv, j, smem_raw, tmem, h, rtile, (int)blockIdx.z,
                          (int)gridDim.z);
  cta_tmem_free(tmem);
}

// Persistent form of the passes over few columns or few rows (projection, survivor
// maintenance, new baselines), for grids of many row tiles, in two kernels.
// pairs_classify: one thread per row of every unit (a 128-row tile of one head); the
// rows of units without any column (projection at r* = 0 mod 128, survivor maintenance
// without evictions) are finished there without TMEM, and every unit with work is
// appended to w.loop_list.  tc_pairs_loop: 2 CTAs per SM take those units one at a time
// from a counter and run the tensor pipeline on each, TMEM allocated once per CTA; the
// units are taken as the CTAs free up, so heads of different budgets (rows of 2,340 to
// 18,720 columns) spread evenly.  In a step whose layers admit nothing almost no unit has
// work, and a launch of one CTA per unit would spend its time starting CTAs.
// Work list and counters of a persistent pass (projection 0, survivors 1, new baselines 2).
template <int MODE>
__host__ __device__ __forceinline__ int loop_slot() {
  return MODE == TM_PROJECT ? 0 : (MODE == TM_SUB ? 1 : 2);
}

template <int MODE, int P>
__global__ void __launch_bounds__(256) pairs_classify(TcJob j, int n_units) {
  int32_t* list = j.w.loop_list + loop_slot<MODE>() * j.w.loop_stride;
  int32_t* ctr = j.w.loop_ctr + 2 * loop_slot<MODE>();
  const int64_t total = (int64_t)n_units * BM;
  for (int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; idx < total;
       idx += (int64_t)gridDim.x * blockDim.x) {
    const int u = (int)(idx / BM), rr = (int)(idx % BM);
    int h, rtile;
    unit_of(j, u, h, rtile);
    const DevHead hd = j.w.hd[h];
    int nrows, c0, c1;
    job_range(MODE, hd, *layer_of(j.w, h), nrows, c0, c1);
    const int row = rtile * BM + rr;
    if (row >= nrows) continue;
    if (c1 > c0) {
      if (rr == 0) list[atomicAdd(&ctr[0], 1)] = u;
    } else if (MODE == TM_PROJECT || MODE == TM_SUB) {
      trivial_row<MODE, P>(j, hd, h, row, c0);
    }
  }
}

template <int MODE, int P, bool KV>
__global__ void __launch_bounds__(THREADS, KV ? 1 : 2)
    tc_pairs_loop(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmAx,
                  const __grid_constant__ CUtensorMap tmB, const __grid_constant__ CUtensorMap tmBx,
                  const __grid_constant__ CUtensorMap tmAv, const __grid_constant__ CUtensorMap tmBv, TcJob j) {
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  if ((smem_u32(smem_raw) & 1023u) != 0u) {
    if (threadIdx.x == 0) dev_fail(j.w.L, DEV_INCONSISTENT, 9903);
    return;
  }
  // the unit index taken by thread 0, passed through the split-tile flag word (unused
  // by these passes)
  volatile int* s_unit = reinterpret_cast<volatile int*>(smem_raw + Lay<KV>::FLAG);
  const int32_t* list = j.w.loop_list + loop_slot<MODE>() * j.w.loop_stride;
  int32_t* ctr = j.w.loop_ctr + 2 * loop_slot<MODE>();
  const int count = __ldcg(&ctr[0]);
  uint32_t tmem = 0;
  bool have_tmem = false;
  for (;;) {
    if (threadIdx.x == 0) *s_unit = atomicAdd(&ctr[1], 1);
    __syncthreads();
    const int k = *s_unit;
    __syncthreads();   // every thread has read it before thread 0 takes the next one
    if (k >= count) break;
    int h, rtile;
    unit_of(j, __ldcg(&list[k]), h, rtile);
    if (!have_tmem) {   // once per CTA, at its first unit
      tmem = cta_tmem_alloc(smem_raw + Lay<KV>::BAR);
      have_tmem = true;
    }
    if (!pairs_unit<MODE, P, KV>(tmA, tmAx, tmB, tmBx, tmAv, tmBv, j, smem_raw, tmem, h, rtile, 0, 1)) break;
  }
  if (have_tmem) cta_tmem_free(tmem);
}

// ---------------------------------------------------------------- crossings, two row tiles
// Persistent form of the crossing pass (keys only).  One CTA per SM takes units of two
// row tiles (256 bank rows of one head) at a fixed stride; each column tile of candidates
// is loaded into shared memory once and feeds the MMAs of both row tiles.  The next
// unit's row tiles load into the second row-tile buffer while the current unit's last
// column tiles run, and the barrier phases run on across units (global tile count T), so
// units follow each other without draining the pipeline or starting a CTA.  TMEM: row
// tile r, accumulator b = T & 1 at columns 128 (2 r + b).  Warps: 0 TMA producer, 1 MMA
// issuer, 2-9 the epilogue of row tile 0 and 10-17 that of row tile 1, each as in the
// one-row-tile form (warps w and w + 4 share TMEM lanes 32 (w % 4) .. +31 and take the
// halves of each column tile, exchanging their half totals every tile).
#ifndef DKV_CROSS_DUAL
#define DKV_CROSS_DUAL 1
#endif
constexpr int DU_EPI = 16;
constexpr int DU_THREADS = 64 + 32 * DU_EPI;
constexpr uint32_t DU_TMEM_COLS = 512;
// Column-tile stages == accumulators: then one barrier per stage can stand for both "the
// tile landed" and "its accumulator is free" (the producer re-arms stage T & 1 only after
// the MMAs of tile T - 2, which waited for that barrier's previous phase).  With more
// stages than accumulators the producer could arm a phase that is still open.
constexpr int DU_STAGES = 2;

struct LayC {
  static constexpr int TILE = 2 * HALF_BYTES;                 // one 128 x 128 bf16 tile
  static constexpr int A = 0;                                 // [2 buffers][2 row tiles]
  static constexpr int B = 4 * TILE;                          // [DU_STAGES] column tiles
  static constexpr int AX = B + DU_STAGES * TILE;             // [2][2] row-form extensions
  static constexpr int BX = AX + 4 * EXT_BYTES;               // [DU_STAGES] column-form
  static constexpr int XCH = BX + DU_STAGES * EXT_BYTES;      // float [2 r][2 b][2 half][BM]
  static constexpr int BAR = XCH + 2 * 2 * 2 * BM * 4;
  // a_full[2] a_free[2] empty[DU_STAGES] rdy[DU_STAGES] accf[2 r][2 b], then the TMEM
  // holder and the abort flag
  static constexpr int NBAR = 2 + 2 + 2 * DU_STAGES + 4;
  static constexpr size_t SMEM = BAR + NBAR * 8 + 16;
  static_assert(B % 1024 == 0 && AX % 1024 == 0, "128-byte-swizzled tiles need 1024-byte alignment");
  static_assert(SMEM <= 227 * 1024, "shared memory per CTA");
};

// Unit u: head h, first row tile rt0 (even) of the pairs of 128-row tiles of each head's
// budget, the pass's rows and columns.  False if the unit has no row.
__device__ __forceinline__ bool cross_unit(const TcJob& j, int u, int& h, int& rt0, int& nrows, int& c0, int& c1) {
  h = j.w.pair_head[u];
  rt0 = 2 * (u - j.w.pair_first[h]);
  job_range(TM_CROSS, j.w.hd[h], *layer_of(j.w, h), nrows, c0, c1);
  return rt0 * BM < nrows;
}

template <int P>
__global__ void __launch_bounds__(DU_THREADS, 1)
    tc_cross_dual(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmAx,
                  const __grid_constant__ CUtensorMap tmB, const __grid_constant__ CUtensorMap tmBx, TcJob j,
                  int n_units) {
  extern __shared__ __align__(1024) uint8_t smem[];
  if ((smem_u32(smem) & 1023u) != 0u) {
    if (threadIdx.x == 0) dev_fail(j.w.L, DEV_INCONSISTENT, 9904);
    return;
  }
  using LY = LayC;
  float* xch = reinterpret_cast<float*>(smem + LY::XCH);
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + LY::BAR);
  uint64_t* a_full = bars + 0;                   // [2] row tiles of a unit landed
  uint64_t* a_free = bars + 2;                   // [2] MMAs of the buffer's last unit complete
  uint64_t* bar_empty = bars + 4;                // [DU_STAGES] MMAs of the stage's tile complete
  uint64_t* bar_rdy = bar_empty + DU_STAGES;     // [DU_STAGES] column tile T landed (stage T & 1)
                                                 //   and accumulator T & 1 released by all 16
                                                 //   epilogue warps: the issuer's one wait per tile
  uint64_t* bar_accf = bar_rdy + DU_STAGES;      // [2 r][2 b] MMAs of row tile r into b complete
  uint32_t* tmem_holder = reinterpret_cast<uint32_t*>(bars + LY::NBAR);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_holder + 1);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    for (int i = 0; i < 2; ++i) {
      mbar_init(a_full + i, 1);
      mbar_init(a_free + i, 1);
    }
    for (int s = 0; s < DU_STAGES; ++s) {
      mbar_init(bar_empty + s, 1);
      mbar_init(bar_rdy + s, DU_EPI + 1);   // the epilogue warps + the producer (with bytes)
    }
    for (int i = 0; i < 4; ++i) mbar_init(bar_accf + i, 1);
    *abort_flag = 0;
    fence_barrier_init();
  }
  if (warp == 1) tmem_alloc(tmem_holder, DU_TMEM_COLS);
  fence_before_sync();
  __syncthreads();
  fence_after_sync();
  const uint32_t tmem = *tmem_holder;

  if (warp == 0) {
    if (lane == 0) {
      // ---------------- TMA producer
      prefetch_map(&tmA); prefetch_map(&tmAx); prefetch_map(&tmB); prefetch_map(&tmBx);
      int k = 0;          // units with columns so far (row-tile buffer k & 1)
      uint32_t T = 0;     // column tiles so far
      bool ok = true;
      for (int u = blockIdx.x; ok && u < n_units; u += gridDim.x) {
        int h, rt0, nrows, c0, c1;
        if (!cross_unit(j, u, h, rt0, nrows, c0, c1) || c1 <= c0) continue;
        const int nt = (c1 - c0 + BN - 1) / BN;
        const int a = k & 1;
        const bool two = (rt0 + 1) * BM < nrows;
        if (!(ok = mbar_wait(a_free + a, ((k >> 1) & 1) ^ 1, abort_flag))) break;
        mbar_arrive_expect_tx(a_full + a, (two ? 2u : 1u) * (uint32_t)(LY::TILE + EXT_BYTES));
        for (int r = 0; r < (two ? 2 : 1); ++r) {
          for (int pn = 0; pn < 2; ++pn)
            tma_load_3d(smem + LY::A + (2 * a + r) * LY::TILE + pn * HALF_BYTES, &tmA, a_full + a, pn * 64,
                        (rt0 + r) * BM, h);
          tma_load_3d(smem + LY::AX + (2 * a + r) * EXT_BYTES, &tmAx, a_full + a, 0, (rt0 + r) * BM, h);
        }
        for (int t = 0; t < nt; ++t, ++T) {
          const int s = (int)(T & 1);
          if (!(ok = mbar_wait(bar_empty + s, ((T >> 1) & 1) ^ 1, abort_flag))) break;
          mbar_arrive_expect_tx(bar_rdy + s, LY::TILE + EXT_BYTES);
          const int col = c0 + t * BN;
          for (int pn = 0; pn < 2; ++pn)
            tma_load_3d(smem + LY::B + s * LY::TILE + pn * HALF_BYTES, &tmB, bar_rdy + s, pn * 64, col, h);
          tma_load_3d(smem + LY::BX + s * EXT_BYTES, &tmBx, bar_rdy + s, 16, col, h);
        }
        ++k;
      }
      if (!ok) {
        *abort_flag = 1;
        dev_fail(j.w.L, DEV_TIMEOUT, 130);
        // copies may still be in flight and nothing will consume them: wait a fixed 50 us,
        // far longer than any copy takes to land
        const uint64_t t0 = globaltimer_ns();
        while (globaltimer_ns() - t0 < 50000ull) {
        }
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      // ---------------- MMA issuer: per column tile 9 MMAs for each row tile (8 k-steps
      // of the keys + 1 of the extension), one wait
      constexpr uint32_t idesc = idesc_bf16(BM, BN);
      const uint64_t bd0 = desc_sw128(smem_u32(smem + LY::B));
      const uint64_t bxd0 = desc_sw32(smem_u32(smem + LY::BX));
      int k = 0;
      uint32_t T = 0;
      bool ok = true, any = false;
      for (int u = blockIdx.x; ok && u < n_units; u += gridDim.x) {
        int h, rt0, nrows, c0, c1;
        if (!cross_unit(j, u, h, rt0, nrows, c0, c1) || c1 <= c0) continue;
        const int nt = (c1 - c0 + BN - 1) / BN;
        const int a = k & 1;
        const bool two = (rt0 + 1) * BM < nrows;
        if (!(ok = mbar_wait(a_full + a, (k >> 1) & 1, abort_flag))) break;
        const uint64_t ad0 = desc_sw128(smem_u32(smem + LY::A + 2 * a * LY::TILE));
        const uint64_t axd0 = desc_sw32(smem_u32(smem + LY::AX + 2 * a * EXT_BYTES));
        for (int t = 0; t < nt; ++t, ++T) {
          const int b = (int)(T & 1);   // stage and accumulator
          if (!(ok = mbar_wait(bar_rdy + b, (T >> 1) & 1, abort_flag))) break;
          fence_after_sync();
          const uint64_t bd = desc_add(bd0, b * LY::TILE);
#pragma unroll
          for (int r = 0; r < 2; ++r) {
            if (r == 0 || two) {
              const uint64_t ad = desc_add(ad0, r * LY::TILE);
              const uint32_t acc = tmem + (uint32_t)((2 * r + b) * BN);
#pragma unroll
              for (int kk = 0; kk < 8; ++kk) {
                const uint32_t koff = (kk >> 2) * HALF_BYTES + (kk & 3) * 32;
                mma_bf16(acc, desc_add(ad, koff), desc_add(bd, koff), idesc, kk > 0);
              }
              mma_bf16(acc, desc_add(axd0, r * EXT_BYTES), desc_add(bxd0, b * EXT_BYTES), idesc, 1u);
            }
            mma_commit(bar_accf + 2 * r + b);   // (no new MMA for an absent row tile: arrives at once)
          }
          mma_commit(bar_empty + b);
          any = true;
        }
        if (!ok) break;
        mma_commit(a_free + a);
        ++k;
      }
      if (!ok) {
        *abort_flag = 1;
        dev_fail(j.w.L, DEV_TIMEOUT, 230);
      }
      // every issued MMA complete before TMEM is freed: a last commit covers all of them
      if (any) {
        mma_commit(a_free + (k & 1));
        volatile int no_abort = 0;
        mbar_wait(a_free + (k & 1), (k >> 1) & 1, &no_abort);
      }
    }
  } else {
    // ---------------- epilogue: thread = row (TMEM lane) of row tile r
    const int ew = warp - 2;                      // 0..15
    const int r = ew >> 3;                        // row tile of the unit
    const int half = (ew >> 2) & 1;               // columns [64 half, 64 half + 64) of each tile
    const int q = warp & 3;                       // TMEM lane quarter
    const int r_local = q * 32 + lane;
    const int bar_id = 1 + q + 4 * r;             // the two warps of this (row tile, quarter)
    const KParams kp = j.kp;
    const float c = pow_c<P>(kp);                 // (sigma^2 / 2)^p
    const uint32_t lane_base = tmem + ((uint32_t)(q * 32) << 16) + (uint32_t)(2 * r * BN);
    float* xr = xch + r * (2 * 2 * BM);           // this row tile's exchange slots [b][half][BM]
    // both accumulators start free: this warp's release for tiles 0 and 1
    if (lane == 0) {
      mbar_arrive(bar_rdy + 0);
      mbar_arrive(bar_rdy + 1);
    }
    uint32_t T = 0;
    bool ok = true;
    // after a failed wait the warp keeps walking every unit and tile without work: the
    // two warps of a row quarter must meet at the same named barriers
    for (int u = blockIdx.x; u < n_units; u += gridDim.x) {
      int h, rt0, nrows, c0, c1;
      if (!cross_unit(j, u, h, rt0, nrows, c0, c1)) continue;
      const int nt = c1 > c0 ? (c1 - c0 + BN - 1) / BN : 0;
      const int row = (rt0 + r) * BM + r_local;
      const bool active = row < nrows;
      const bool tile_live = (rt0 + r) * BM < nrows;   // warp-uniform: the row tile has MMAs
      const int64_t bh = (int64_t)h * j.b.M_max;
      // per-row state (sums in units of |A|^-p)
      float S = 0.f, thr = 0.f;
      int cross = INT_MAX;
      float* snap_row = nullptr;
      if (active) {
        const float rho = j.b.rho[bh + row];
        thr = (__fmul_rn(kp.tau, j.b.base[bh + row]) - rho) / c;
        if (thr <= 0.f) cross = 0;
        snap_row = j.w.snap + (bh + row) * j.w.snap_stride;
        if (half == 0) snap_row[0] = 0.f;
      }
      for (int t = 0; t < nt; ++t, ++T) {
        const int b = (int)(T & 1);
        const int col0 = c0 + t * BN;
        const int nc = min(BN, c1 - col0);
        // every warp waits for the MMAs of its row tile (also an absent one: its release
        // of accumulator b must not run ahead of tile T)
        if (ok) ok = __all_sync(0xffffffffu, mbar_wait(bar_accf + 2 * r + b, (T >> 1) & 1, abort_flag));
        if (!ok) *abort_flag = 1;
        fence_after_sync();
        // chunk totals of this warp's half, then the running sum of the row
        float tot[2] = {0.f, 0.f};
        if (ok && tile_live) {
#pragma unroll
          for (int ch = 0; ch < 2; ++ch) {
            const int cs = half * 64 + ch * 32;
            if (cs >= nc) continue;   // warp-uniform
            float v[32];
            tmem_ld32(lane_base + b * BN + cs, v);
            tmem_wait_ld();
            const int lim = min(32, nc - cs);
            tot[ch] = lim == 32 ? chunk_sum<P>(v) : chunk_sum_partial<P>(v, lim);
          }
        }
        // exchange the half totals of this row, so both warps carry the same running sum
        const float mine = tot[0] + tot[1];
        xr[(b * 2 + half) * BM + r_local] = mine;
        named_bar(bar_id, 64);
        const float other = xr[(b * 2 + (half ^ 1)) * BM + r_local];
        const float T0 = half == 0 ? mine : other;
        const float T1 = half == 0 ? other : mine;
        const float base0 = half == 0 ? S : S + T0;
        int hit = -1;
        float run = base0;
        if (ok && active && cross == INT_MAX) {
          if (base0 + tot[0] >= thr) hit = 0;
          else if ((base0 + tot[0]) + tot[1] >= thr) { hit = 1; run = base0 + tot[0]; }
        }
        // exact position inside the chunk, term by term (at most once per row); the TMEM
        // load is warp-collective, so the whole warp takes part for each chunk hit
#pragma unroll
        for (int hc = 0; hc < 2; ++hc) {
          const int cs = half * 64 + hc * 32;
          if (cs < nc && __any_sync(0xffffffffu, hit == hc)) {
            float v[32];
            tmem_ld32(lane_base + b * BN + cs, v);
            tmem_wait_ld();
            if (hit == hc) {
              const int lim = min(32, nc - cs);
              // the 32 terms are independent: all of them first (in place), then the
              // running sum
#pragma unroll
              for (int jj = 0; jj < 32; ++jj) v[jj] = term1<P>(v[jj]);
              int pos = lim;
#pragma unroll
              for (int jj = 0; jj < 32; ++jj) {
                if (jj < lim && pos == lim) {
                  run += v[jj];
                  if (run >= thr) pos = jj + 1;
                }
              }
              cross = col0 + cs + pos;
            }
          }
        }
        S = (S + T0) + T1;
        if (ok && active && half == 0 && nc == BN) snap_row[(col0 + BN) / SNAP] = S;
        if (ok) {
          fence_before_sync();
          __syncwarp();
          if (lane == 0) mbar_arrive(bar_rdy + b);   // accumulator b free for tile T + 2
        }
      }
      // unit end: each half saw only its own columns, the row's first crossing is the
      // earlier one.  The exchange slots of accumulator T & 1 were last read before the
      // barrier of tile T - 1; a second barrier keeps the next unit's first tile from
      // writing them before the partner warp has read.
      int* xi = reinterpret_cast<int*>(xr + (T & 1) * 2 * BM);
      xi[half * BM + r_local] = cross;
      named_bar(bar_id, 64);
      cross = min(xi[r_local], xi[BM + r_local]);
      named_bar(bar_id, 64);
      if (ok && active && half == 0) {
        const DevLayer L = *layer_of(j.w, h);
        j.w.cross[bh + row] = cross;
        const int bin = cross == INT_MAX ? L.rmax + 1 : cross;
        atomicAdd(&j.w.hist[(int64_t)h * j.w.hist_stride + bin], 1);
      }
    }
    if (!ok) {
      *abort_flag = 1;
      if (lane == 0) dev_fail(j.w.L, DEV_TIMEOUT, 330);
    }
  }
  fence_before_sync();
  __syncthreads();
  if (warp == 1) {
    fence_after_sync();
    tmem_dealloc(tmem, DU_TMEM_COLS);
  }
}

// ---------------------------------------------------------------- scores, 256-column tiles
// Persistent form of the score pass (keys only) for grids of many candidate row tiles.
// One CTA per SM takes candidate row tiles (units) at a fixed stride; each bank tile of
// 256 columns is one MMA instruction per k-step (N = 256), so the row tile is read from
// shared memory once per 256 columns instead of once per 128 and the issuing thread has
// half the instructions per FLOP.  TMEM: two accumulators of 256 columns (all 512).  The
// next unit's row tile loads into the second row-tile buffer during the current unit and
// barrier phases run on across units (global tile count T).  Warps: 0 TMA producer, 1
// MMA issuer, 2-17 the epilogue: warp w takes TMEM lane quarter w % 4 and the 64-column
// quarter (w - 2) / 4 of each tile, in the 16x256b layout of the one-row-tile form.
#ifndef DKV_SCORE_WIDE
#define DKV_SCORE_WIDE 1
#endif
constexpr int SW_BN = 256;                         // columns per tile
constexpr int SW_EPI = 16;
constexpr int SW_THREADS = 64 + 32 * SW_EPI;
constexpr int SW_STAGES = 2;                       // == accumulators (one barrier per stage)
constexpr int SW_META = SW_STAGES + 3;             // weights ring (the argument of META_BUFS)
constexpr int SW_APANEL = BM * 128;                // 64-column panel of the 128-row tile (16 KiB)
constexpr int SW_BPANEL = SW_BN * 128;             // 64-column panel of the 256-row tile (32 KiB)
constexpr int SW_BEXT = SW_BN * 32;                // 256 extension rows (8 KiB)

struct LayW {
  static constexpr int A = 0;                                    // [2 buffers][2 panels]
  static constexpr int B = 2 * 2 * SW_APANEL;                    // [SW_STAGES][2 panels]
  static constexpr int AX = B + SW_STAGES * 2 * SW_BPANEL;       // [2] row-form extensions
  static constexpr int BX = AX + 2 * EXT_BYTES;                  // [SW_STAGES] column-form
  static constexpr int META = BX + SW_STAGES * SW_BEXT;          // float [SW_META][SW_BN]
  static constexpr int XF = META + SW_META * SW_BN * 4;          // float [4 column quarters][BM]
  static constexpr int BAR = XF + 4 * BM * 4;
  // a_full[2] a_free[2] empty[S] rdy[S] accf[2] meta[SW_META], then the TMEM holder and
  // the abort flag
  static constexpr int NBAR = 2 + 2 + 2 * SW_STAGES + 2 + SW_META;
  static constexpr size_t SMEM = BAR + NBAR * 8 + 16;
  static_assert(B % 1024 == 0 && AX % 1024 == 0 && BX % 256 == 0, "swizzled tiles need aligned bases");
  static_assert(SMEM <= 227 * 1024, "shared memory per CTA");
};

// Unit u: candidate row tile u % tpn of the (u / tpn)-th head in order of decreasing
// budget (the largest units first: the fixed stride then ends on small ones); the pass's
// rows and bank columns.  False if the unit has no row.
__device__ __forceinline__ bool wide_unit(const TcJob& j, int u, int& h, int& rt, int& nrows, int& c0, int& c1) {
  h = j.w.head_order[u / j.tpn];
  rt = u % j.tpn;
  job_range(TM_SCORE, j.w.hd[h], *layer_of(j.w, h), nrows, c0, c1);
  return rt * BM < nrows && c1 > c0;
}

template <int P>
__global__ void __launch_bounds__(SW_THREADS, 1)
    tc_score_wide(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmAx,
                  const __grid_constant__ CUtensorMap tmB, const __grid_constant__ CUtensorMap tmBx, TcJob j,
                  int n_units) {
  extern __shared__ __align__(1024) uint8_t smem[];
  if ((smem_u32(smem) & 1023u) != 0u) {
    if (threadIdx.x == 0) dev_fail(j.w.L, DEV_INCONSISTENT, 9906);
    return;
  }
  using LY = LayW;
  float* meta = reinterpret_cast<float*>(smem + LY::META);
  float* xf = reinterpret_cast<float*>(smem + LY::XF);
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + LY::BAR);
  uint64_t* a_full = bars + 0;                   // [2] row tile of a unit landed
  uint64_t* a_free = bars + 2;                   // [2] MMAs of the buffer's last unit complete
  uint64_t* bar_empty = bars + 4;                // [S] MMAs of the stage's tile complete
  uint64_t* bar_rdy = bar_empty + SW_STAGES;     // [S] bank tile T landed (stage T & 1) and
                                                 //   accumulator T & 1 released by all 16 warps
  uint64_t* bar_accf = bar_rdy + SW_STAGES;      // [2] MMAs into the accumulator complete
  uint64_t* bar_meta = bar_accf + 2;             // [SW_META] weights of tile T
  uint32_t* tmem_holder = reinterpret_cast<uint32_t*>(bars + LY::NBAR);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_holder + 1);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    for (int i = 0; i < 2; ++i) {
      mbar_init(a_full + i, 1);
      mbar_init(a_free + i, 1);
      mbar_init(bar_accf + i, 1);
    }
    for (int s = 0; s < SW_STAGES; ++s) {
      mbar_init(bar_empty + s, 1);
      mbar_init(bar_rdy + s, SW_EPI + 1);   // the epilogue warps + the producer (with bytes)
    }
    for (int q = 0; q < SW_META; ++q) mbar_init(bar_meta + q, 1);
    *abort_flag = 0;
    fence_barrier_init();
  }
  if (warp == 1) tmem_alloc(tmem_holder, DU_TMEM_COLS);
  fence_before_sync();
  __syncthreads();
  fence_after_sync();
  const uint32_t tmem = *tmem_holder;

  if (warp == 0) {
    if (lane == 0) {
      // ---------------- TMA producer
      prefetch_map(&tmA); prefetch_map(&tmAx); prefetch_map(&tmB); prefetch_map(&tmBx);
      int k = 0;
      uint32_t T = 0;
      bool ok = true;
      for (int u = blockIdx.x; ok && u < n_units; u += gridDim.x) {
        int h, rt, nrows, c0, c1;
        if (!wide_unit(j, u, h, rt, nrows, c0, c1)) continue;
        const int nt = (c1 - c0 + SW_BN - 1) / SW_BN;
        const int a = k & 1;
        if (!(ok = mbar_wait(a_free + a, ((k >> 1) & 1) ^ 1, abort_flag))) break;
        mbar_arrive_expect_tx(a_full + a, 2 * SW_APANEL + EXT_BYTES);
        for (int pn = 0; pn < 2; ++pn)
          tma_load_3d(smem + LY::A + (2 * a + pn) * SW_APANEL, &tmA, a_full + a, pn * 64, rt * BM, h);
        tma_load_3d(smem + LY::AX + a * EXT_BYTES, &tmAx, a_full + a, 0, rt * BM, h);
        for (int t = 0; t < nt; ++t, ++T) {
          const int s = (int)(T & 1);
          if (!(ok = mbar_wait(bar_empty + s, ((T >> 1) & 1) ^ 1, abort_flag))) break;
          mbar_arrive_expect_tx(bar_rdy + s, 2 * SW_BPANEL + SW_BEXT);
          const int col = c0 + t * SW_BN;
          for (int pn = 0; pn < 2; ++pn)
            tma_load_3d(smem + LY::B + (2 * s + pn) * SW_BPANEL, &tmB, bar_rdy + s, pn * 64, col, h);
          tma_load_3d(smem + LY::BX + s * SW_BEXT, &tmBx, bar_rdy + s, 16, col, h);
          const int q = (int)(T % SW_META);
          mbar_arrive_expect_tx(bar_meta + q, SW_BN * 4);
          bulk_load(meta + q * SW_BN, j.w.invb + (int64_t)h * j.w.invb_stride + col, SW_BN * 4, bar_meta + q);
        }
        ++k;
      }
      if (!ok) {
        *abort_flag = 1;
        dev_fail(j.w.L, DEV_TIMEOUT, 150);
        const uint64_t t0 = globaltimer_ns();   // copies may still land: a fixed 50 us
        while (globaltimer_ns() - t0 < 50000ull) {
        }
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      // ---------------- MMA issuer: per bank tile 8 k-steps of N = 256 + 1 of the extension
      constexpr uint32_t idesc = idesc_bf16(BM, SW_BN);
      const uint64_t bd0 = desc_sw128(smem_u32(smem + LY::B));
      const uint64_t bxd0 = desc_sw32(smem_u32(smem + LY::BX));
      int k = 0;
      uint32_t T = 0;
      bool ok = true, any = false;
      for (int u = blockIdx.x; ok && u < n_units; u += gridDim.x) {
        int h, rt, nrows, c0, c1;
        if (!wide_unit(j, u, h, rt, nrows, c0, c1)) continue;
        const int nt = (c1 - c0 + SW_BN - 1) / SW_BN;
        const int a = k & 1;
        if (!(ok = mbar_wait(a_full + a, (k >> 1) & 1, abort_flag))) break;
        const uint64_t ad = desc_sw128(smem_u32(smem + LY::A + 2 * a * SW_APANEL));
        const uint64_t axd = desc_sw32(smem_u32(smem + LY::AX + a * EXT_BYTES));
        for (int t = 0; t < nt; ++t, ++T) {
          const int b = (int)(T & 1);   // stage and accumulator
          if (!(ok = mbar_wait(bar_rdy + b, (T >> 1) & 1, abort_flag))) break;
          fence_after_sync();
          const uint64_t bd = desc_add(bd0, 2 * b * SW_BPANEL);
          const uint32_t acc = tmem + (uint32_t)(b * SW_BN);
#pragma unroll
          for (int kk = 0; kk < 8; ++kk)
            mma_bf16(acc, desc_add(ad, (kk >> 2) * SW_APANEL + (kk & 3) * 32),
                     desc_add(bd, (kk >> 2) * SW_BPANEL + (kk & 3) * 32), idesc, kk > 0);
          mma_bf16(acc, axd, desc_add(bxd0, b * SW_BEXT), idesc, 1u);
          mma_commit(bar_accf + b);
          mma_commit(bar_empty + b);
          any = true;
        }
        if (!ok) break;
        mma_commit(a_free + a);
        ++k;
      }
      if (!ok) {
        *abort_flag = 1;
        dev_fail(j.w.L, DEV_TIMEOUT, 250);
      }
      if (any) {   // every issued MMA complete before TMEM is freed
        mma_commit(a_free + (k & 1));
        volatile int no_abort = 0;
        mbar_wait(a_free + (k & 1), (k >> 1) & 1, &no_abort);
      }
    }
  } else {
    // ---------------- epilogue: lane quarter q, columns [64 cq, 64 cq + 64) of each tile
    const int ew = warp - 2;                      // 0..15
    const int cq = ew >> 2;                       // column quarter
    const int q = warp & 3;                       // TMEM lane quarter
    const int r_local = q * 32 + lane;
    const int bar_id = 1 + q;                     // the four warps of this lane quarter
    const float c = pow_c<P>(j.kp);
    const uint32_t lane_base = tmem + ((uint32_t)(q * 32) << 16);
    if (lane == 0) {   // both accumulators start free: this warp's release for tiles 0 and 1
      mbar_arrive(bar_rdy + 0);
      mbar_arrive(bar_rdy + 1);
    }
    uint32_t T = 0;
    bool ok = true;
    // after a failed wait the warp keeps walking every unit and tile without work: the
    // four warps of a lane quarter must meet at the same named barriers
    for (int u = blockIdx.x; u < n_units; u += gridDim.x) {
      int h, rt, nrows, c0, c1;
      if (!wide_unit(j, u, h, rt, nrows, c0, c1)) continue;
      const int nt = (c1 - c0 + SW_BN - 1) / SW_BN;
      float2 sacc[4];   // rows lane/4 + 8 jj of the quarter (16x256b layout)
#pragma unroll
      for (int jj = 0; jj < 4; ++jj) sacc[jj] = make_float2(0.f, 0.f);
      for (int t = 0; t < nt; ++t, ++T) {
        const int b = (int)(T & 1);
        const int col0 = c0 + t * SW_BN;
        const int nc = min(SW_BN, c1 - col0);
        if (ok) ok = __all_sync(0xffffffffu, mbar_wait(bar_accf + b, (T >> 1) & 1, abort_flag));
        if (ok) ok = __all_sync(0xffffffffu, mbar_wait(bar_meta + T % SW_META, (T / SW_META) & 1, abort_flag));
        if (!ok) {
          *abort_flag = 1;
          continue;
        }
        fence_after_sync();
        const int cs = 64 * cq;
        if (cs < nc) {   // warp-uniform
          float va[32], vb[32];
          tmem_ld16x256b_x8(lane_base + b * SW_BN + cs, va);
          tmem_ld16x256b_x8(lane_base + (16u << 16) + b * SW_BN + cs, vb);
          tmem_wait_ld();
          fence_before_sync();
          __syncwarp();
          if (lane == 0) mbar_arrive(bar_rdy + b);   // accumulator b free for tile T + 2
          score_rows4<P>(va, vb, meta + (T % SW_META) * SW_BN + cs, nc - cs, 2 * (lane & 3), sacc);
        } else {
          fence_before_sync();
          __syncwarp();
          if (lane == 0) mbar_arrive(bar_rdy + b);
        }
      }
      // unit end: the four column quarters of each row, added in quarter order; a second
      // barrier keeps the next unit's sums from being written before every warp has read
#pragma unroll
      for (int jj = 0; jj < 4; ++jj) {
        float x = sacc[jj].x + sacc[jj].y;
        x += __shfl_xor_sync(0xffffffffu, x, 1);
        x += __shfl_xor_sync(0xffffffffu, x, 2);
        if ((lane & 3) == 0) xf[cq * BM + q * 32 + (lane >> 2) + 8 * jj] = P == 1 ? -x : x;
      }
      named_bar(bar_id, 128);
      const float acc = ((xf[r_local] + xf[BM + r_local]) + xf[2 * BM + r_local]) + xf[3 * BM + r_local];
      named_bar(bar_id, 128);
      const int row = rt * BM + r_local;
      if (ok && cq == 0 && row < nrows)
        j.w.score[(int64_t)h * j.b.n_max + row] = (acc * c) / (float)j.w.hd[h].m_old;
    }
    if (!ok && lane == 0) dev_fail(j.w.L, DEV_TIMEOUT, 350);
  }
  fence_before_sync();
  __syncthreads();
  if (warp == 1) {
    fence_after_sync();
    tmem_dealloc(tmem, DU_TMEM_COLS);
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

bool encode(CUtensorMap* m, const void* base, uint64_t inner, int64_t rows, int64_t heads, uint32_t box_inner,
            uint32_t box_rows, CUtensorMapSwizzle sw) {
  EncodeTiledFn fn = encode_fn();
  if (!fn || rows < 1 || heads < 1) return false;
  cuuint64_t dims[3] = {inner, (cuuint64_t)rows, (cuuint64_t)heads};
  cuuint64_t strides[2] = {inner * 2, (cuuint64_t)rows * inner * 2};
  cuuint32_t box[3] = {box_inner, box_rows, 1};
  cuuint32_t es[3] = {1, 1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides, box, es,
            CU_TENSOR_MAP_INTERLEAVE_NONE, sw, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

}  // namespace

// bf16 [heads][rows][128] keys: boxes of 64 columns x box_rows rows, 128-byte swizzle.
bool make_map_rows(CUtensorMap* m, const void* base, int64_t rows, int64_t heads, int box_rows) {
  return encode(m, base, 128, rows, heads, 64, box_rows, CU_TENSOR_MAP_SWIZZLE_128B);
}

// bf16 [heads][rows][32] extension rows: boxes of 16 columns x box_rows rows, 32-byte swizzle.
bool make_map_ext(CUtensorMap* m, const void* base, int64_t rows, int64_t heads, int box_rows) {
  return encode(m, base, 32, rows, heads, 16, box_rows, CU_TENSOR_MAP_SWIZZLE_32B);
}

namespace {

template <int MODE, int P>
void launch_p(dim3 grid, cudaStream_t s, const CUtensorMap& a, const CUtensorMap& ax, const CUtensorMap& b,
              const CUtensorMap& bx, const CUtensorMap& av, const CUtensorMap& bv, bool kv, const TcJob& job,
              int n_units) {
  if (n_units > 0) {   // persistent form (projection, survivor maintenance, new baselines)
    if constexpr (MODE == TM_PROJECT || MODE == TM_SUB || MODE == TM_NEWBASE) {
      if (cudaMemsetAsync(job.w.loop_ctr + 2 * loop_slot<MODE>(), 0, 2 * sizeof(int32_t), s) != cudaSuccess) return;
      const int64_t threads = (int64_t)n_units * BM;
      const int cblocks = (int)std::min<int64_t>((threads + 255) / 256, (int64_t)grid.x * 8);
      pairs_classify<MODE, P><<<cblocks, 256, 0, s>>>(job, n_units);
      if (kv) tc_pairs_loop<MODE, P, true><<<grid, THREADS, Lay<true>::SMEM, s>>>(a, ax, b, bx, av, bv, job);
      else tc_pairs_loop<MODE, P, false><<<grid, THREADS, Lay<false>::SMEM, s>>>(a, ax, b, bx, av, bv, job);
    }
    return;
  }
  if (kv) tc_pairs<MODE, P, true><<<grid, THREADS, Lay<true>::SMEM, s>>>(a, ax, b, bx, av, bv, job);
  else tc_pairs<MODE, P, false><<<grid, THREADS, Lay<false>::SMEM, s>>>(a, ax, b, bx, av, bv, job);
}

// rv / cv: the row and column values (same layouts as rk / ck), non-null only with the
// [K; V] descriptor; the extension rows rx / cx then carry the descriptors' norms.
template <int MODE>
cudaError_t launch_tc(const Bank& b, const Ws& w, const KParams& kp, const void* rk, const void* rx, int64_t rk_rows,
                      const void* ck, const void* cx, int64_t ck_rows, int max_rows, cudaStream_t s, Timer* t,
                      const char* name, int split = 1, const void* rv = nullptr, const void* cv = nullptr,
                      int64_t rx_rows = 0) {
  const bool kv = rv != nullptr;
  CUtensorMap ma, max_, mb, mbx, mav, mbv;
  if (!make_map_rows(&ma, rk, rk_rows, b.H, BM) || !make_map_ext(&max_, rx, rx_rows > 0 ? rx_rows : rk_rows, b.H, BM) ||
      !make_map_rows(&mb, ck, ck_rows, b.H, BN) || !make_map_ext(&mbx, cx, ck_rows, b.H, BN))
    return cudaErrorInvalidValue;
  if (kv) {
    if (!cv || !make_map_rows(&mav, rv, rk_rows, b.H, BM) || !make_map_rows(&mbv, cv, ck_rows, b.H, BN))
      return cudaErrorInvalidValue;
  } else {
    mav = ma;   // never read
    mbv = mb;
  }
  const int n_sm = sm_count();
  if constexpr (MODE == TM_CROSS) {
    if (DKV_CROSS_DUAL && !kv && n_sm > 0) {   // the persistent two-row-tile form
      TcJob job{b, w, kp, 0, 0};
      timer_begin(t, name, s);
      if (kp.p == 1) tc_cross_dual<1><<<n_sm, DU_THREADS, LayC::SMEM, s>>>(ma, max_, mb, mbx, job, w.n_mpairs);
      else if (kp.p == 4) tc_cross_dual<4><<<n_sm, DU_THREADS, LayC::SMEM, s>>>(ma, max_, mb, mbx, job, w.n_mpairs);
      else tc_cross_dual<2><<<n_sm, DU_THREADS, LayC::SMEM, s>>>(ma, max_, mb, mbx, job, w.n_mpairs);
      timer_end(t, s);
      return cudaGetLastError();
    }
  }
  // passes over bank rows take one CTA per budget-sized row tile of each head
  const int lin = (MODE == TM_CROSS || MODE == TM_PROJECT || MODE == TM_SUB) && split == 1 ? 1 : 0;
  const int tpn = (max_rows + BM - 1) / BM;
  TcJob job{b, w, kp, lin, tpn};
  dim3 grid(lin ? w.n_mtiles : tpn, lin ? 1 : b.H, split);
  // projection, survivor maintenance and new baselines over many row tiles: the
  // persistent form, a few CTAs per SM (most of those row tiles have no column when
  // layers admit nothing)
  int n_units = 0;
  if ((MODE == TM_PROJECT || MODE == TM_SUB || MODE == TM_NEWBASE) && n_sm > 0) {
    const int units = lin ? w.n_mtiles : tpn * b.H;
    if (units >= 16 * n_sm) {
      n_units = units;
      grid = dim3((kv ? 1 : 2) * n_sm, 1, 1);
    }
  }
  timer_begin(t, name, s);
  if (kp.p == 1) launch_p<MODE, 1>(grid, s, ma, max_, mb, mbx, mav, mbv, kv, job, n_units);
  else if (kp.p == 4) launch_p<MODE, 4>(grid, s, ma, max_, mb, mbx, mav, mbv, kv, job, n_units);
  else launch_p<MODE, 2>(grid, s, ma, max_, mb, mbx, mav, mbv, kv, job, n_units);
  timer_end(t, s);
  return cudaGetLastError();
}

}  // namespace

bool tc_supported(int d, int bf16) { return d == 128 && bf16 && encode_fn() != nullptr; }

int sm_count() {
  static int n = 0;
  if (n == 0) {
    int dev = 0, v = 0;
    if (cudaGetDevice(&dev) == cudaSuccess && cudaDeviceGetAttribute(&v, cudaDevAttrMultiProcessorCount, dev) == cudaSuccess)
      n = v;
  }
  return n;
}

cudaError_t tc_attn_set_smem_limits();

cudaError_t tc_set_smem_limits() {
  cudaError_t e = cudaSuccess;
#define DKV_OPT1(M, P, KV)                                                                                     \
  if (e == cudaSuccess)                                                                                        \
    e = cudaFuncSetAttribute(tc_pairs<M, P, KV>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)Lay<KV>::SMEM);
#define DKV_OPTL(M, P, KV)                                                                                     \
  if (e == cudaSuccess)                                                                                        \
    e = cudaFuncSetAttribute(tc_pairs_loop<M, P, KV>, cudaFuncAttributeMaxDynamicSharedMemorySize,             \
                             (int)Lay<KV>::SMEM);
#define DKV_OPT(M)                                                                                             \
  DKV_OPT1(M, 1, false) DKV_OPT1(M, 2, false) DKV_OPT1(M, 4, false)                                            \
  DKV_OPT1(M, 1, true) DKV_OPT1(M, 2, true) DKV_OPT1(M, 4, true)
#define DKV_OPTLOOP(M)                                                                                         \
  DKV_OPTL(M, 1, false) DKV_OPTL(M, 2, false) DKV_OPTL(M, 4, false)                                            \
  DKV_OPTL(M, 1, true) DKV_OPTL(M, 2, true) DKV_OPTL(M, 4, true)
  DKV_OPT(TM_SCORE)
  DKV_OPT(TM_CROSS)
  DKV_OPT(TM_PROJECT)
  DKV_OPT(TM_SUB)
  DKV_OPT(TM_NEWBASE)
  DKV_OPTLOOP(TM_PROJECT)
  DKV_OPTLOOP(TM_SUB)
  DKV_OPTLOOP(TM_NEWBASE)
#define DKV_OPTD(P)                                                                                           \
  if (e == cudaSuccess)                                                                                        \
    e = cudaFuncSetAttribute(tc_cross_dual<P>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)LayC::SMEM);
  DKV_OPTD(1) DKV_OPTD(2) DKV_OPTD(4)
#undef DKV_OPTD
#define DKV_OPTW(P)                                                                                           \
  if (e == cudaSuccess)                                                                                        \
    e = cudaFuncSetAttribute(tc_score_wide<P>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)LayW::SMEM);
  DKV_OPTW(1) DKV_OPTW(2) DKV_OPTW(4)
#undef DKV_OPTW
#undef DKV_OPTLOOP
#undef DKV_OPTL
#undef DKV_OPT
#undef DKV_OPT1
  if (e == cudaSuccess) e = tc_attn_set_smem_limits();
  return e;
}

// With the [K; V] descriptor every pass also reads the values beside its keys (same
// sources as the fp32 passes: the candidates' values, vperm, the bank's, vsurv, vevict).
#ifndef DKV_SCORE_SPLIT
#define DKV_SCORE_SPLIT 0   // 0: by grid size, else the split itself
#endif

cudaError_t launch_score_tc(const Bank& b, const Ws& w, const void* Kc, const void* Vc, int N, const KParams& kp,
                            cudaStream_t s, Timer* t) {
  const bool kv = w.vperm != nullptr;
  // the candidates (caller's array) are [H][N][d]; their extension rows, like every
  // candidate array of the workspace, [H][n_max][32].  The bank columns are split over two
  // CTAs per row tile while the row tiles alone would not fill the GPU several times over
  int split = DKV_SCORE_SPLIT;
  const int n_sm = sm_count();
  const int64_t ctas = (int64_t)((N + BM - 1) / BM) * b.H;
  if (split == 0) split = n_sm > 0 && ctas >= 16 * (int64_t)n_sm ? 1 : 2;
  if (DKV_SCORE_WIDE && split == 1 && !kv && n_sm > 0) {
    // the persistent 256-column form over the many row tiles
    CUtensorMap ma, max_, mb, mbx;
    if (!make_map_rows(&ma, Kc, N, b.H, BM) || !make_map_ext(&max_, w.cext, b.n_max, b.H, BM) ||
        !make_map_rows(&mb, b.k, b.M_max, b.H, SW_BN) || !make_map_ext(&mbx, w.bext, b.M_max, b.H, SW_BN))
      return cudaErrorInvalidValue;
    const int tpn = (N + BM - 1) / BM;
    TcJob job{b, w, kp, 0, tpn};
    const int n_units = (int)ctas;
    timer_begin(t, "score_tc", s);
    if (kp.p == 1) tc_score_wide<1><<<n_sm, SW_THREADS, LayW::SMEM, s>>>(ma, max_, mb, mbx, job, n_units);
    else if (kp.p == 4) tc_score_wide<4><<<n_sm, SW_THREADS, LayW::SMEM, s>>>(ma, max_, mb, mbx, job, n_units);
    else tc_score_wide<2><<<n_sm, SW_THREADS, LayW::SMEM, s>>>(ma, max_, mb, mbx, job, n_units);
    timer_end(t, s);
    return cudaGetLastError();
  }
  return launch_tc<TM_SCORE>(b, w, kp, Kc, w.cext, N, b.k, w.bext, b.M_max, N, s, t, "score_tc", split,
                             kv ? Vc : nullptr, kv ? b.v : nullptr, b.n_max);
}

cudaError_t launch_cross_tc(const Bank& b, const Ws& w, const KParams& kp, cudaStream_t s, Timer* t) {
  const bool kv = w.vperm != nullptr;
  return launch_tc<TM_CROSS>(b, w, kp, b.k, w.bext, b.M_max, w.kperm, w.kperm_ext, b.n_max, b.M_max, s, t,
                             "cross_tc", 1, kv ? b.v : nullptr, w.vperm);
}

cudaError_t launch_project_tc(const Bank& b, const Ws& w, const KParams& kp, cudaStream_t s, Timer* t) {
  const bool kv = w.vperm != nullptr;
  return launch_tc<TM_PROJECT>(b, w, kp, b.k, w.bext, b.M_max, w.kperm, w.kperm_ext, b.n_max, b.M_max, s, t,
                               "project_tc", 1, kv ? b.v : nullptr, w.vperm);
}

cudaError_t launch_subtract_tc(const Bank& b, const Ws& w, const KParams& kp, cudaStream_t s, Timer* t) {
  return launch_tc<TM_SUB>(b, w, kp, w.ksurv, w.ksurv_ext, b.M_max, w.kevict, w.kevict_ext, b.n_max, b.M_max, s,
                           t, "subtract_tc", 1, w.vsurv, w.vevict);
}

cudaError_t launch_newbase_tc(const Bank& b, const Ws& w, const KParams& kp, cudaStream_t s, Timer* t) {
  const bool kv = w.vperm != nullptr;
  return launch_tc<TM_NEWBASE>(b, w, kp, w.kperm, w.kperm_ext, b.n_max, b.k, w.bext, b.M_max, b.n_max, s, t,
                               "newbase_tc", 2, w.vperm, kv ? b.v : nullptr);
}

}  // namespace dkv
