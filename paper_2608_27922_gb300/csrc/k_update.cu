// Selection, ordering and compaction kernels of the bank update (no pair math).
//
//   cand_norms   ||k_x||^2 of the candidates (fp32) and their extension rows, plus (one
//                extra block) the snapshot of occupancy, budgets and prefix range; with
//                temporal re-zeroing (App. A) the keys are first rotated back to temporal
//                rotary coordinate 0 and stored, and the norms taken of the stored keys
//   sort         stable ascending order of the Eq. 6 scores, ties by source index (Alg. 1),
//                and the candidate keys copied into that order (operand of the prefix passes)
//   rstar_*      violator counts c_r = #{cross <= r}, budgets e_r (Eq. 10), feasibility,
//                and the largest prefix feasible for every head (Eq. 11)
//   select       mandatory set {g(r*) >= tau} plus the densest rho~(r*) (Step 3), via a
//                radix select on the fp32 bit patterns; ties evict the older state
//   commit       Eq. 12: admitted keys/values into the evicted slots, the rest appended;
//                keys of the surviving and of the evicted states copied out first
//                (operands of Eq. C.4)
#include "dkv.h"
#include "dkv_internal.h"

#include <algorithm>

#include <climits>

namespace dkv {

namespace {

constexpr int BIG = 1024;   // threads of the one-block-per-head kernels

__device__ __forceinline__ int warp_id() { return threadIdx.x >> 5; }
__device__ __forceinline__ int lane_id() { return threadIdx.x & 31; }

// Row copies as a flat loop over groups of four 16-byte chunks (64 bytes) of a row.
// Every row is a whole number of groups and no group spans two sources, so a thread
// resolves its row once and has four independent loads in flight before its stores.
// map(row, group) returns the group's source and destination (src == nullptr: nothing
// to copy) and performs the row's scalar updates for one of its groups.
struct Group4 {
  const uint4* src;
  uint4* dst;
};

template <typename Map>
__device__ __forceinline__ void copy_groups(int nrows, int per_row, Map map) {
  const int total = nrows * per_row;
  for (int c = blockIdx.x * blockDim.x + threadIdx.x; c < total; c += gridDim.x * blockDim.x) {
    const int row = c / per_row, grp = c - row * per_row;
    const Group4 g = map(row, grp);
    if (g.src) {
      uint4 v[4];
#pragma unroll
      for (int k = 0; k < 4; ++k) v[k] = g.src[k];
#pragma unroll
      for (int k = 0; k < 4; ++k) g.dst[k] = v[k];
    }
  }
}

// One 64-byte group: all four loads are issued before the stores.
__device__ __forceinline__ void copy64(const uint4* src, uint4* dst) {
  uint4 v[4];
#pragma unroll
  for (int k = 0; k < 4; ++k) v[k] = src[k];
#pragma unroll
  for (int k = 0; k < 4; ++k) dst[k] = v[k];
}

// Snapshot of occupancy and budgets per head and the prefix range of this update,
// per layer (one block): rmax = min(N, min over the layer's live heads of M_h).
__device__ __forceinline__ void prepare_body(const Bank& b, const Ws& w, int N, int64_t step) {
  const int G = b.H / w.layer_heads;
  // per layer, until the last phase: rmax holds the minimum budget of its live heads and
  // empty_all their count
  for (int g = threadIdx.x; g < G; g += blockDim.x) {
    DevLayer* L = w.L + g;
    L->N = N;
    L->step = step;
    L->r_star = 0;
    L->rmax = INT_MAX;
    L->empty_all = 0;
  }
  __syncthreads();
  for (int h = threadIdx.x; h < b.H; h += blockDim.x) {
    int m = b.occ[h];
    const int M = w.budgets[h];
    if (m < 0 || m > M) {
      dev_fail(w.L, DEV_INCONSISTENT, 1000 + h);
      m = m < 0 ? 0 : M;
    }
    DevHead hd;
    hd.m_old = m; hd.M = M; hd.r = 0; hd.e = 0; hd.n_mand = 0; hd.n_pre = 0; hd.m_new = m;
    hd.empty = (m == 0);
    w.hd[h] = hd;
    if (m > 0) {
      DevLayer* L = layer_of(w, h);
      atomicMin(&L->rmax, M);
      atomicAdd(&L->empty_all, 1);
    }
  }
  __syncthreads();
  for (int g = threadIdx.x; g < G; g += blockDim.x) {
    DevLayer* L = w.L + g;
    const int live = __ldcg(&L->empty_all), min_budget = __ldcg(&L->rmax);
    L->empty_all = live == 0;
    L->rmax = live ? min(N, min_budget) : 0;
  }
}

// bf16 split x = hi + mid + lo (each rounded to nearest), ~24 significant bits.
__device__ __forceinline__ void split3(float x, __nv_bfloat16& hi, __nv_bfloat16& mid, __nv_bfloat16& lo) {
  hi = __float2bfloat16_rn(x);
  const float r1 = x - __bfloat162float(hi);
  mid = __float2bfloat16_rn(r1);
  lo = __float2bfloat16_rn(r1 - __bfloat162float(mid));
}

// Sum of squares of the pl (2 or 4) consecutive elements at p, one vector load.
template <typename T>
__device__ __forceinline__ float sq_sum(const T* p, int pl) {
  float x[4];
  if constexpr (sizeof(T) == 2) {
    if (pl == 4) {
      const uint2 u = *reinterpret_cast<const uint2*>(p);
      const __nv_bfloat162 a = *reinterpret_cast<const __nv_bfloat162*>(&u.x);
      const __nv_bfloat162 c = *reinterpret_cast<const __nv_bfloat162*>(&u.y);
      x[0] = __low2float(a); x[1] = __high2float(a); x[2] = __low2float(c); x[3] = __high2float(c);
    } else {
      const __nv_bfloat162 a = *reinterpret_cast<const __nv_bfloat162*>(p);
      x[0] = __low2float(a); x[1] = __high2float(a); x[2] = 0.f; x[3] = 0.f;
    }
  } else {
    if (pl == 4) {
      const float4 f = *reinterpret_cast<const float4*>(p);
      x[0] = f.x; x[1] = f.y; x[2] = f.z; x[3] = f.w;
    } else {
      const float2 f = *reinterpret_cast<const float2*>(p);
      x[0] = f.x; x[1] = f.y; x[2] = 0.f; x[3] = 0.f;
    }
  }
  return fmaf(x[3], x[3], fmaf(x[2], x[2], fmaf(x[1], x[1], x[0] * x[0])));
}

// ||k||^2 per row and, if ext != nullptr, the row's 32 extension values used by the
// tensor-core passes: row form [-g_hi, -g_mid, -g_lo, 1, 1, 1, 0 x 10] and column form
// [1, 1, 1, -h_hi, -h_mid, -h_lo, 0 x 10], g = |k|^2 / 2 + goff, h = |k|^2 / 2.
// A warp takes NR_ROWS rows (lane = d / 32 consecutive elements of each, one vector load),
// with all loads issued before the reductions.
constexpr int NR_ROWS = 4;

// Warp reduction of the lanes' partial squares a[q] of rows row0 + q (< n), then the
// norm and (ext != nullptr) the extension row of each.
__device__ __forceinline__ void norms_ext_tail(float* a, int h, int row0, int n, float* __restrict__ out,
                                               int64_t out_hs, __nv_bfloat16* __restrict__ ext, int64_t ext_hs,
                                               float goff) {
  const int l = lane_id();
#pragma unroll
  for (int q = 0; q < NR_ROWS; ++q)
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) a[q] += __shfl_xor_sync(0xffffffffu, a[q], o);
#pragma unroll
  for (int q = 0; q < NR_ROWS; ++q) {
    const int row = row0 + q;
    if (row >= n) break;
    if (l == 0) out[(int64_t)h * out_hs + row] = a[q];
    if (ext) {
      __nv_bfloat16 g[3], hh[3];
      split3(-(0.5f * a[q] + goff), g[0], g[1], g[2]);
      split3(-(0.5f * a[q]), hh[0], hh[1], hh[2]);
      const __nv_bfloat16 one = __float2bfloat16_rn(1.0f), zero = __float2bfloat16_rn(0.0f);
      __nv_bfloat16 v = zero;
      if (l < 3) v = g[l];
      else if (l < 6) v = one;
      else if (l >= 16 && l < 19) v = one;
      else if (l >= 19 && l < 22) v = hh[l - 19];
      ext[(int64_t)h * ext_hs + (int64_t)row * 32 + l] = v;
    }
  }
}

// V != nullptr ([K; V] descriptor): the norms are those of [k; v], V laid out like K.
template <typename T>
__device__ __forceinline__ void row_norms_body(const T* __restrict__ K, const T* __restrict__ V, int64_t head_stride,
                                               int rows_cap, const int32_t* count, int count_is_occ, int N,
                                               float* __restrict__ out, int64_t out_hs, int d,
                                               __nv_bfloat16* __restrict__ ext, int64_t ext_hs, float goff) {
  const int h = blockIdx.y;
  const int row0 = (blockIdx.x * (blockDim.x / 32) + warp_id()) * NR_ROWS;
  const int n = min(count_is_occ ? count[h] : N, rows_cap);
  if (row0 >= n) return;
  const int pl = d / 32;
  const int l = lane_id();
  float a[NR_ROWS];
#pragma unroll
  for (int q = 0; q < NR_ROWS; ++q) {
    const int64_t off = (int64_t)h * head_stride + (int64_t)(row0 + q) * d + l * pl;
    a[q] = row0 + q < n ? sq_sum<T>(K + off, pl) : 0.f;
    if (V && row0 + q < n) a[q] += sq_sum<T>(V + off, pl);
  }
  norms_ext_tail(a, h, row0, n, out, out_hs, ext, ext_hs, goff);
}

// ---- temporal rotary re-zeroing (App. A: memory keys carry temporal coordinate 0) ----
// A rotation pair (x, y) of a key rotated by a = t theta (t the token's temporal
// coordinate) is moved back by -a:  x0 = x cos a + y sin a,  y0 = y cos a - x sin a,
// i.e. rot(u, v) = u cos a + v sin a with (u, v) = (x, y) and (y, -x).  The stored value is
// the nearest value of the key's type (ties to even) to the exact rotation.
//
// cos a and sin a come from a per-CTA table: float64 sincos of the exact float64 angle,
// once per distinct coordinate among the CTA's rows and pair (not per element or head).
// bf16 keys: r = u c + v s in fp32 with c, s the table values rounded to fp32
// (|c - cos a|, |s - sin a| <= 2^-24.99), so |r - exact| <= 2^-24 (|u| + 2 |v| + |r|) < E.
// Rounding is monotone: when both ends of [r - E, r + E] (rounded outwards) give the
// same bf16 value, that is the rounding of the exact rotation; otherwise (about 1
// element in 2,000) r is taken in float64 from the float64 table.  fp32 keys: float64.

// float64 evaluation rounded once to the key type: bf16 through float32 rounded to odd
// (exact for a later rounding to 8 significant bits).
template <typename T>
__device__ __forceinline__ float rot_f64(float u, float v, double c, double s) {
  const double r = (double)u * c + (double)v * s;
  if constexpr (sizeof(T) == 4) {
    return __double2float_rn(r);
  } else {
    float f = __double2float_rz(r);
    if ((double)f != r) f = __uint_as_float(__float_as_uint(f) | 1u);
    return __bfloat162float(__float2bfloat16_rn(f));
  }
}

template <typename T>
__device__ __forceinline__ float rot_tab(float u, float v, float c, float s, double cd, double sd) {
  if constexpr (sizeof(T) == 2) {
    const float r = fmaf(u, c, v * s);
    const float E = 0x1p-23f * (fabsf(u) + fabsf(v) + fabsf(r)) + 0x1p-126f;
    const __nv_bfloat16 lo = __float2bfloat16_rn(__fsub_rd(r, E));
    const __nv_bfloat16 hi = __float2bfloat16_rn(__fadd_ru(r, E));
    if (__bfloat16_as_ushort(lo) == __bfloat16_as_ushort(hi)) return __bfloat162float(lo);
  }
  return rot_f64<T>(u, v, cd, sd);
}

template <typename T>
__device__ __forceinline__ void load_lane(const T* p, int pl, float* x) {
  if constexpr (sizeof(T) == 2) {
    if (pl == 4) {
      const uint2 u = *reinterpret_cast<const uint2*>(p);
      const __nv_bfloat162 a = *reinterpret_cast<const __nv_bfloat162*>(&u.x);
      const __nv_bfloat162 c = *reinterpret_cast<const __nv_bfloat162*>(&u.y);
      x[0] = __low2float(a); x[1] = __high2float(a); x[2] = __low2float(c); x[3] = __high2float(c);
    } else {
      const __nv_bfloat162 a = *reinterpret_cast<const __nv_bfloat162*>(p);
      x[0] = __low2float(a); x[1] = __high2float(a); x[2] = 0.f; x[3] = 0.f;
    }
  } else {
    if (pl == 4) {
      const float4 f = *reinterpret_cast<const float4*>(p);
      x[0] = f.x; x[1] = f.y; x[2] = f.z; x[3] = f.w;
    } else {
      const float2 f = *reinterpret_cast<const float2*>(p);
      x[0] = f.x; x[1] = f.y; x[2] = 0.f; x[3] = 0.f;
    }
  }
}

// Stores values that are exactly representable in T.
template <typename T>
__device__ __forceinline__ void store_lane(T* p, int pl, const float* x) {
  if constexpr (sizeof(T) == 2) {
    const __nv_bfloat162 a = __floats2bfloat162_rn(x[0], x[1]);
    if (pl == 4) {
      const __nv_bfloat162 c = __floats2bfloat162_rn(x[2], x[3]);
      uint2 u;
      u.x = *reinterpret_cast<const uint32_t*>(&a);
      u.y = *reinterpret_cast<const uint32_t*>(&c);
      *reinterpret_cast<uint2*>(p) = u;
    } else {
      *reinterpret_cast<__nv_bfloat162*>(p) = a;
    }
  } else {
    if (pl == 4) *reinterpret_cast<float4*>(p) = make_float4(x[0], x[1], x[2], x[3]);
    else *reinterpret_cast<float2*>(p) = make_float2(x[0], x[1]);
  }
}

constexpr int ROPE_ROWS = 8;   // candidate rows per CTA of the re-zeroing prepare (all heads)

struct RopeTab {
  float th[64];                    // theta_j
  int t[ROPE_ROWS];                // temporal coordinate of each row
  int lead[ROPE_ROWS];             // first row of the CTA with the same coordinate
  float cf[ROPE_ROWS][64], sf[ROPE_ROWS][64];     // cos / sin rounded to fp32 (leader rows)
  double cd[ROPE_ROWS][64], sd[ROPE_ROWS][64];    // cos / sin in float64
};

// The lane's pl elements (from element e0 of a row of the CTA's table row q) rotated back.
// Interleaved layout: the lane holds whole pairs.  Half layout: the partner of element e
// is e +- d/2, held by lane l ^ 16 at the same position (called by all 32 lanes).
template <typename T>
__device__ __forceinline__ void rope_lane(float* x, int pl, int e0, int d, int layout, const RopeTab& tb, int q) {
  const int t = tb.t[q];
  const int k = tb.lead[q];
  if (layout == 0) {
#pragma unroll
    for (int i = 0; i < 4; i += 2) {
      if (i >= pl) break;
      const int j = (e0 + i) >> 1;
      if (tb.th[j] == 0.f || t == 0) continue;
      const float u = x[i], v = x[i + 1];
      x[i] = rot_tab<T>(u, v, tb.cf[k][j], tb.sf[k][j], tb.cd[k][j], tb.sd[k][j]);
      x[i + 1] = rot_tab<T>(v, -u, tb.cf[k][j], tb.sf[k][j], tb.cd[k][j], tb.sd[k][j]);
    }
  } else {
    const int half = d / 2;
    const bool first = e0 < half;
    float o[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) o[i] = __shfl_xor_sync(0xffffffffu, x[i], 16);
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      if (i >= pl) break;
      const int j = (e0 + i) % half;
      if (tb.th[j] == 0.f || t == 0) continue;
      x[i] = rot_tab<T>(x[i], first ? o[i] : -o[i], tb.cf[k][j], tb.sf[k][j], tb.cd[k][j], tb.sd[k][j]);
    }
  }
}

template <typename T>
__global__ void k_row_norms(const T* __restrict__ K, const T* __restrict__ V, int64_t head_stride, int rows_cap,
                            const int32_t* count, int count_is_occ, int N, float* __restrict__ out, int64_t out_hs,
                            int d, __nv_bfloat16* __restrict__ ext, int64_t ext_hs, float goff) {
  row_norms_body<T>(K, V, head_stride, rows_cap, count, count_is_occ, N, out, out_hs, d, ext, ext_hs, goff);
}

// First kernel of an update: the candidates' norms and extension rows, the zeroed
// crossing histogram, and the update snapshot (prepare_body) in one extra block (last x,
// head 0); the three share no data.
template <typename T>
__global__ void k_cand_prepare(Bank b, Ws w, const T* __restrict__ Kc, const T* __restrict__ Vc, int N, int64_t step,
                               float goff) {
  if (blockIdx.x == gridDim.x - 1) {
    if (blockIdx.y == 0) prepare_body(b, w, N, step);
    return;
  }
  {
    const int64_t nh = (int64_t)b.H * w.hist_stride;
    const int64_t nthr = (int64_t)(gridDim.x - 1) * gridDim.y * blockDim.x;
    for (int64_t i = ((int64_t)blockIdx.y * (gridDim.x - 1) + blockIdx.x) * blockDim.x + threadIdx.x; i < nh;
         i += nthr)
      w.hist[i] = 0;
  }
  row_norms_body<T>(Kc, Vc, (int64_t)N * b.d, N, nullptr, 0, N, w.cnorm, b.n_max, b.d, (__nv_bfloat16*)w.cext,
                    (int64_t)b.n_max * 32, goff);
}

// k_cand_prepare with temporal re-zeroing: CTA x takes candidate rows [8x, 8x + 8) of every
// head.  It builds the cos / sin table of its rows' distinct coordinates, then its warps
// take batches of NR_ROWS rows of one head: rotated back into w.kevict ([H][N][d], the
// layout of Kc), norms and extension rows of the stored keys.  Last CTA: prepare_body.
template <typename T>
__global__ void __launch_bounds__(256) k_cand_prepare_rope(Bank b, Ws w, const T* __restrict__ Kc,
                                                           const T* __restrict__ Vc, int N, int64_t step, float goff,
                                                           const RopeArgs ra) {
  if (blockIdx.x == gridDim.x - 1) {
    prepare_body(b, w, N, step);
    return;
  }
  {
    const int64_t nh = (int64_t)b.H * w.hist_stride;
    const int64_t nthr = (int64_t)(gridDim.x - 1) * blockDim.x;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < nh; i += nthr) w.hist[i] = 0;
  }
  __shared__ RopeTab tb;
  const int d = b.d, P = d / 2;
  const int x0 = blockIdx.x * ROPE_ROWS;
  const int nr = min(ROPE_ROWS, N - x0);
  if (threadIdx.x < P) tb.th[threadIdx.x] = __ldg(ra.theta + threadIdx.x);
  if (threadIdx.x < nr) tb.t[threadIdx.x] = __ldg(ra.tpos + x0 + threadIdx.x);
  __syncthreads();
  if (threadIdx.x < nr) {
    int k = threadIdx.x;
    for (int q = 0; q < (int)threadIdx.x; ++q)
      if (tb.t[q] == tb.t[threadIdx.x]) { k = q; break; }
    tb.lead[threadIdx.x] = k;
  }
  __syncthreads();
  for (int i = threadIdx.x; i < nr * P; i += blockDim.x) {
    const int q = i / P, j = i % P;
    if (tb.lead[q] != q) continue;
    double sv = 0.0, cv = 1.0;
    if (tb.th[j] != 0.f && tb.t[q] != 0) sincos((double)tb.t[q] * (double)tb.th[j], &sv, &cv);
    tb.cd[q][j] = cv;
    tb.sd[q][j] = sv;
    tb.cf[q][j] = (float)cv;
    tb.sf[q][j] = (float)sv;
  }
  __syncthreads();
  T* __restrict__ Kout = (T*)w.kevict;
  const int pl = d / 32, l = lane_id();
  const int nw = blockDim.x / 32;
  for (int base = warp_id() * NR_ROWS; base < b.H * ROPE_ROWS; base += nw * NR_ROWS) {
    const int h = base / ROPE_ROWS, q0 = base % ROPE_ROWS;   // NR_ROWS divides ROPE_ROWS: one head
    if (q0 >= nr) continue;                                    // warp-uniform
    float x[NR_ROWS][4];
#pragma unroll
    for (int q = 0; q < NR_ROWS; ++q)
      if (q0 + q < nr) load_lane<T>(Kc + ((int64_t)h * N + x0 + q0 + q) * d + l * pl, pl, x[q]);
    float a[NR_ROWS];
#pragma unroll
    for (int q = 0; q < NR_ROWS; ++q) {
      a[q] = 0.f;
      if (q0 + q >= nr) continue;                              // warp-uniform
      rope_lane<T>(x[q], pl, l * pl, d, ra.layout, tb, q0 + q);
      store_lane<T>(Kout + ((int64_t)h * N + x0 + q0 + q) * d + l * pl, pl, x[q]);
      a[q] = fmaf(x[q][3], x[q][3], fmaf(x[q][2], x[q][2], fmaf(x[q][1], x[q][1], x[q][0] * x[q][0])));
      if (Vc) a[q] += sq_sum<T>(Vc + ((int64_t)h * N + x0 + q0 + q) * d + l * pl, pl);   // [K; V] descriptor
    }
    norms_ext_tail(a, h, x0 + q0, x0 + nr, w.cnorm, b.n_max, (__nv_bfloat16*)w.cext, (int64_t)b.n_max * 32, goff);
  }
}

// Sort of the keys (fkey(score) << 32 | source index) per head: ascending score, equal
// scores in source order (the keys are unique, so any correct sort is the stable one).
// Phase 1 sorts runs of RUN = 256 keys, one warp each, with a bitonic network kept in
// registers (thread = SKPT consecutive keys; strides below SKPT) and warp shuffles
// (longer strides).  Phase 2 places every key at its index in its own run plus its
// rank in each other run, so no merge levels are needed and every run is placed by
// its own block.
constexpr int SKPT = 8;
constexpr int RUN = 32 * SKPT;

template <int J>
__device__ __forceinline__ void cas_regs_c(unsigned long long (&x)[SKPT], int t, int k) {
#pragma unroll
  for (int r = 0; r < SKPT; ++r) {
    if ((r ^ J) > r) {
      const int i = t * SKPT + r;
      const bool up = (i & k) == 0;
      const unsigned long long a = x[r], c = x[r ^ J];
      if ((a > c) == up) { x[r] = c; x[r ^ J] = a; }
    }
  }
}

// in-register compare-exchange at stride j < SKPT (strides as compile-time constants)
__device__ __forceinline__ void cas_regs(unsigned long long (&x)[SKPT], int t, int k, int j) {
  if (j == 4) cas_regs_c<4>(x, t, k);
  else if (j == 2) cas_regs_c<2>(x, t, k);
  else cas_regs_c<1>(x, t, k);
}

// compare-exchange with the lane at distance j / SKPT
__device__ __forceinline__ void cas_shfl(unsigned long long (&x)[SKPT], int t, int k, int j) {
  const int ld = j / SKPT;
  const bool lower = (t & ld) == 0;   // this lane holds the lower element of each pair
#pragma unroll
  for (int r = 0; r < SKPT; ++r) {
    const unsigned long long o = __shfl_xor_sync(0xffffffffu, x[r], ld);
    const int i = t * SKPT + r;
    const bool up = (i & k) == 0;
    const unsigned long long lo = x[r] < o ? x[r] : o, hi = x[r] < o ? o : x[r];
    x[r] = (lower == up) ? lo : hi;
  }
}

// Phase 1: warp w of block x sorts run a = 8 x + w (source indices [256 a, 256 a + 256),
// padded with ~0) ascending; the direction bit is taken from the run-local index, so
// every run comes out ascending.
__global__ void __launch_bounds__(256) k_sort_runs(Ws w, int n_max, int identity) {
  const int h = blockIdx.y;
  const int N = layer_of(w, h)->N;
  // empty bank: source order (Alg. 1, m = 0 branch); source-order policy: the same
  if (w.hd[h].empty || identity) {
    for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < N; i += gridDim.x * blockDim.x)
      w.perm[(int64_t)h * n_max + i] = i;
    return;
  }
  const int a = blockIdx.x * 8 + warp_id();
  if (a * RUN >= N) return;                       // warp-uniform
  const int t = lane_id();
  const float* sc = w.score + (int64_t)h * n_max;
  unsigned long long x[SKPT];
#pragma unroll
  for (int r = 0; r < SKPT; ++r) {
    const int i = a * RUN + t * SKPT + r;
    x[r] = i < N ? ((unsigned long long)fkey(sc[i]) << 32) | (unsigned)i : ~0ull;
  }
  for (int k = 2; k <= RUN; k <<= 1)
    for (int j = k >> 1; j > 0; j >>= 1) {
      if (j < SKPT) cas_regs(x, t, k, j);
      else cas_shfl(x, t, k, j);
    }
  unsigned long long* out = w.sortbuf + (int64_t)h * w.sort_stride + a * RUN + t * SKPT;
#pragma unroll
  for (int r = 0; r < SKPT; r += 2)
    *reinterpret_cast<ulonglong2*>(out + r) = make_ulonglong2(x[r], x[r + 1]);
}

// Number of keys of the sorted run r[0..RUN) below x (branchless, 9 probes).
__device__ __forceinline__ int run_rank(const unsigned long long* r, unsigned long long x) {
  int pos = 0;
#pragma unroll
  for (int s = RUN / 2; s > 0; s >>= 1)
    if (r[pos + s - 1] < x) pos += s;
  return pos + (r[pos] < x ? 1 : 0);
}

// Phase 2: block (a, h) places the keys of runs RB a .. RB a + RB - 1: final position =
// index in its run plus the number of smaller keys in every other run (keys are unique,
// so positions are distinct and cover [0, N)).  The block then copies its candidates'
// keys, norms and extension rows to their positions (the operand of the prefix passes in
// pi order).
// Source order (empty bank, or the source-order policy): position = source index.
template <int RB>
__global__ void __launch_bounds__(RUN * RB) k_sort_rank(Bank bk, Ws w, const char* __restrict__ Kc,
                                                        const char* __restrict__ Vc, int esize, int identity) {
  extern __shared__ unsigned long long runs[];
  __shared__ int s_pos[RUN * RB], s_src[RUN * RB];
  const int h = blockIdx.y;
  const int N = layer_of(w, h)->N;
  const int64_t hn = (int64_t)h * bk.n_max;
  const int nruns = (N + RUN - 1) / RUN;
  const int a0 = blockIdx.x * RB;
  if (a0 >= nruns) return;                        // block-uniform
  const int t = threadIdx.x;
  const int a = a0 + t / RUN, tr = t % RUN;       // this thread's run and key within it
  const bool ident = w.hd[h].empty || identity;
  if (ident) {
    s_pos[t] = s_src[t] = a * RUN + tr;           // rows past N are skipped below
  } else {
    const unsigned long long* src = w.sortbuf + (int64_t)h * w.sort_stride;
    for (int i = t; i < nruns * RUN / 2; i += RUN * RB)
      reinterpret_cast<ulonglong2*>(runs)[i] = reinterpret_cast<const ulonglong2*>(src)[i];
    __syncthreads();
    const bool in_run = a < nruns;
    const unsigned long long x = in_run ? runs[a * RUN + tr] : ~0ull;
    const int nvalid = in_run ? min(RUN, N - a * RUN) : 0;   // padding (~0) sorts to the end
    int pos = -1;
    if (tr < nvalid) {
      pos = tr;
      int b = 0;
      for (; b + 4 <= nruns; b += 4) {
        int c[4];
#pragma unroll
        for (int u = 0; u < 4; ++u) c[u] = b + u == a ? 0 : run_rank(runs + (b + u) * RUN, x);
        pos += (c[0] + c[1]) + (c[2] + c[3]);
      }
      for (; b < nruns; ++b)
        if (b != a) pos += run_rank(runs + b * RUN, x);
      if (pos >= N || x == ~0ull) {
        dev_fail(w.L, DEV_INCONSISTENT, 8800 + h);
        pos = -1;
      } else {
        w.perm[hn + pos] = (int32_t)(x & 0xffffffffu);
      }
    }
    s_pos[t] = pos;
    s_src[t] = tr < nvalid ? (int)(x & 0xffffffffu) : -1;
  }
  __syncthreads();
  const int rb = bk.d * esize;
  const int kg = rb / 64;                         // key groups, one extension group, then
  const int vg = w.vperm ? kg : 0;                // value groups ([K; V] descriptor)
  const int per_row = kg + 1 + vg;
  // every reader of the copy takes positions below the layer's rmax (the crossing,
  // projection and new-baseline passes, the commit), or, in an empty bank, below
  // min(N, M_h) (the candidates it admits in source order): later positions are not copied
  const DevHead hd = w.hd[h];
  const int need = hd.empty ? min(N, hd.M) : layer_of(w, h)->rmax;
  for (int c = t; c < RUN * RB * per_row; c += RUN * RB) {
    const int row = c / per_row, grp = c - row * per_row;
    const int pos = s_pos[row], src = s_src[row];
    if (pos < 0 || pos >= need || src < 0 || src >= N) continue;   // not needed, no row, or reported above
    if (grp < kg) {
      copy64(reinterpret_cast<const uint4*>(Kc + ((int64_t)h * N + src) * rb) + 4 * grp,
             reinterpret_cast<uint4*>((char*)w.kperm + (hn + pos) * rb) + 4 * grp);
    } else if (grp > kg) {
      copy64(reinterpret_cast<const uint4*>(Vc + ((int64_t)h * N + src) * rb) + 4 * (grp - kg - 1),
             reinterpret_cast<uint4*>((char*)w.vperm + (hn + pos) * rb) + 4 * (grp - kg - 1));
    } else {
      w.kperm_norm[hn + pos] = w.cnorm[hn + src];
      copy64(reinterpret_cast<const uint4*>((const char*)w.cext + (hn + src) * 64),
             reinterpret_cast<uint4*>((char*)w.kperm_ext + (hn + pos) * 64));
    }
  }
}

// Per head: c_r = #{i : cross_i <= r} and feasibility c_r <= e_r for r in [0, rmax].
// Reads a DevHead written by another block of the same launch (bypassing L1).
__device__ __forceinline__ DevHead ld_head_cg(const DevHead* p) {
  DevHead hd;
  const int4 a = __ldcg(reinterpret_cast<const int4*>(p));
  const int4 c = __ldcg(reinterpret_cast<const int4*>(p) + 1);
  hd.m_old = a.x; hd.M = a.y; hd.r = a.z; hd.e = a.w;
  hd.n_mand = c.x; hd.n_pre = c.y; hd.m_new = c.z; hd.empty = c.w;
  return hd;
}

// One block per head: violator counts c_r (prefix sums of the crossing histogram),
// budgets e_r (Eq. 10) and the feasibility bit of every prefix r; the last block of a
// layer to finish combines that layer's heads (Eq. 11) and sets r, e of each of them.
__global__ void __launch_bounds__(BIG) k_rstar(Bank b, Ws w, int sync_heads) {
  __shared__ int s_tot[BIG];
  __shared__ int s_best, s_last;
  const int h = blockIdx.x;
  const DevHead hd = w.hd[h];
  DevLayer* lay = layer_of(w, h);
  const int rmax = lay->rmax;
  const int N = lay->N;
  const int lh = w.layer_heads;
  const int h0 = h / lh * lh;   // first head of this layer
  uint32_t* feas = w.feas + (int64_t)h * w.feas_words;
  const int nw = (rmax + 1 + 31) / 32;
  if (threadIdx.x == 0) s_best = 0;
  if (hd.empty) {   // an empty head does not constrain the shared prefix
    for (int i = threadIdx.x; i < nw; i += blockDim.x) feas[i] = 0xffffffffu;
  } else {
    for (int i = threadIdx.x; i < nw; i += blockDim.x) feas[i] = 0u;
    const int n = rmax + 1;
    const int chunk = (n + blockDim.x - 1) / blockDim.x;
    const int lo = threadIdx.x * chunk, hi = min(n, lo + chunk);
    const int32_t* hist = w.hist + (int64_t)h * w.hist_stride;
    int tot = 0;
    for (int r = lo; r < hi; ++r) tot += hist[r];
    s_tot[threadIdx.x] = tot;
    __syncthreads();
    for (int o = 1; o < (int)blockDim.x; o <<= 1) {   // inclusive Hillis-Steele scan
      const int v = threadIdx.x >= o ? s_tot[threadIdx.x - o] : 0;
      __syncthreads();
      s_tot[threadIdx.x] += v;
      __syncthreads();
    }
    int c = s_tot[threadIdx.x] - tot;   // exclusive prefix
    int best = 0;
    for (int r = lo; r < hi; ++r) {
      c += hist[r];
      const int e = max(0, hd.m_old + r - hd.M);
      const bool ok = (r == 0) || (c <= e);   // r = 0 is always feasible (Sec. 3.4 Step 2)
      if (ok) {
        atomicOr(&feas[r >> 5], 1u << (r & 31));
        best = r;
      }
    }
    atomicMax(&s_best, best);
  }
  __threadfence();
  __syncthreads();
  if (threadIdx.x == 0) {
    if (!hd.empty) w.hd[h].r = s_best;   // largest feasible prefix of this head alone
    __threadfence();
    s_last = atomicAdd(&lay->arrive, 1) == lh - 1;   // the layer's last head to arrive
  }
  __syncthreads();
  if (!s_last) return;
  // ---- last block: the layer's shared prefix
  __threadfence();
  if (threadIdx.x == 0) s_best = 0;
  __syncthreads();
  if (sync_heads) {
    for (int i = threadIdx.x; i < nw; i += blockDim.x) {
      uint32_t a = 0xffffffffu;
      for (int hh = h0; hh < h0 + lh; ++hh) a &= __ldcg(w.feas + (int64_t)hh * w.feas_words + i);
      if (i == nw - 1 && ((rmax + 1) & 31)) a &= (1u << ((rmax + 1) & 31)) - 1u;
      if (i == 0) a |= 1u;
      if (a) atomicMax(&s_best, i * 32 + 31 - __clz(a));
    }
  }
  __syncthreads();
  const int rstar = s_best;
  __shared__ int s_rmax_used, s_rmin_used;
  if (threadIdx.x == 0) { s_rmax_used = 0; s_rmin_used = INT_MAX; }
  __syncthreads();
  for (int hh = h0 + threadIdx.x; hh < h0 + lh; hh += blockDim.x) {
    DevHead d = ld_head_cg(w.hd + hh);
    int r;
    if (d.empty) r = min(N, d.M);
    else r = sync_heads ? rstar : d.r;
    d.r = r;
    d.e = d.empty ? 0 : max(0, d.m_old + r - d.M);
    w.hd[hh] = d;
    atomicMax(&s_rmax_used, r);
    atomicMin(&s_rmin_used, r);
  }
  __syncthreads();
  // reported r*: Alg. 1's min(N, M) when every head starts empty (min over per-head budgets),
  // the shared prefix when synchronised, else the largest per-head prefix
  if (threadIdx.x == 0) {
    lay->r_star = lay->empty_all ? s_rmin_used : (sync_heads ? rstar : s_rmax_used);
    lay->arrive = 0;
  }
}

// Block-wide exclusive scan of one flag per thread; returns this thread's offset and
// writes the block total to *total.
__device__ int block_scan_flag(int flag, int* s_warp, int* total) {
  const unsigned bal = __ballot_sync(0xffffffffu, flag);
  const int within = __popc(bal & ((1u << lane_id()) - 1u));
  if (lane_id() == 0) s_warp[warp_id()] = __popc(bal);
  __syncthreads();
  if (warp_id() == 0) {   // exclusive scan of the warp counts by one warp
    const int nw = (int)(blockDim.x / 32);
    const int v = lane_id() < nw ? s_warp[lane_id()] : 0;
    int incl = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int x = __shfl_up_sync(0xffffffffu, incl, o);
      if (lane_id() >= o) incl += x;
    }
    if (lane_id() < nw) s_warp[lane_id()] = incl - v;
    if (lane_id() == 31) s_warp[32] = incl;
  }
  __syncthreads();
  const int off = s_warp[warp_id()] + within;
  *total = s_warp[32];
  __syncthreads();
  return off;
}

// Adds one to s_hist[bin] for every lane with valid set, one shared-memory atomic per
// distinct bin of the warp (all 32 lanes must call it).
__device__ __forceinline__ void hist_add(int* s_hist, bool valid, unsigned bin) {
  const unsigned key = valid ? bin : 0xffffffffu;
  const unsigned peers = __match_any_sync(0xffffffffu, key);
  if (valid && lane_id() == __ffs(peers) - 1) atomicAdd(&s_hist[bin], __popc(peers));
}

// Warp 0: the bin of a 256-bin histogram where the running count, taken from the top
// bin down (from_top) or from bin 0 up, first reaches kk (>= 1).  Returns the bin and
// kk minus the count before it through *bin and *rest; false if the total is below kk.
__device__ bool find_bin(const int* s_hist, unsigned kk, bool from_top, unsigned* bin, unsigned* rest) {
  const int l = lane_id();
  unsigned c[8], cnt = 0;
#pragma unroll
  for (int j = 0; j < 8; ++j) {
    const int bj = from_top ? 255 - (8 * l + j) : 8 * l + j;
    c[j] = (unsigned)s_hist[bj];
    cnt += c[j];
  }
  unsigned incl = cnt;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const unsigned v = __shfl_up_sync(0xffffffffu, incl, o);
    if (l >= o) incl += v;
  }
  const unsigned hit = __ballot_sync(0xffffffffu, incl >= kk);
  if (hit == 0u) return false;
  const int src = __ffs(hit) - 1;
  unsigned my_bin = 0, my_rest = 0;
  if (l == src) {
    unsigned cum = incl - cnt;
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      if (cum + c[j] >= kk) {
        my_bin = from_top ? 255 - (8 * l + j) : 8 * l + j;
        my_rest = kk - cum;
        break;
      }
      cum += c[j];
    }
  }
  *bin = __shfl_sync(0xffffffffu, my_bin, src);
  *rest = __shfl_sync(0xffffffffu, my_rest, src);
  return true;
}

// Banks up to SEL_STAGE states are staged in shared memory for the select passes (sort
// key of rho~ and a mandatory bit per state); larger ones are re-read from global memory.
constexpr int SEL_STAGE = 40960;

__host__ __device__ constexpr size_t sel_smem_bytes(int m_cap) {
  return m_cap > SEL_STAGE ? 0 : (size_t)m_cap * 4 + ((size_t)m_cap + 31) / 32 * 4;
}

__global__ void __launch_bounds__(BIG) k_select(Bank b, Ws w, int eviction) {
  extern __shared__ uint32_t s_stage[];   // [m] sort keys, then [(m + 31) / 32] mandatory bits
  __shared__ int s_hist[256];
  __shared__ int s_warp[33];
  __shared__ int s_cnt[2];
  __shared__ unsigned s_prefix, s_kk;
  __shared__ unsigned long long s_tprefix;
  const int h = blockIdx.x;
  const DevHead hd = w.hd[h];
  const int64_t bh = (int64_t)h * b.M_max;
  const int m = hd.m_old;
  const int r = hd.r;
  const int e = hd.e;
  const int32_t* cross = w.cross + bh;
  const float* rt = w.rho_t + bh;
  if (hd.empty) return;
  if (threadIdx.x == 0) { s_cnt[0] = 0; s_cnt[1] = 0; }
  __syncthreads();
  // mandatory set and pre-violators (and the shared-memory stage of keys and flags)
  const bool staged = b.M_max <= SEL_STAGE;
  uint32_t* skey = s_stage;
  uint32_t* smand = s_stage + (staged ? b.M_max : 0);
  int nm = 0, npre = 0;
  for (int base = 0; base < m; base += blockDim.x) {
    const int i = base + threadIdx.x;
    bool mand = false;
    if (i < m) {
      const int c = cross[i];
      npre += (c == 0);
      mand = r > 0 && c <= r;
      nm += mand;
      if (staged) skey[i] = fkey(rt[i]);
    }
    const unsigned bal = __ballot_sync(0xffffffffu, mand);
    if (staged && lane_id() == 0 && i < m) smand[i >> 5] = bal;
  }
  nm = __reduce_add_sync(0xffffffffu, nm);
  npre = __reduce_add_sync(0xffffffffu, npre);
  if (lane_id() == 0) {
    atomicAdd(&s_cnt[0], nm);
    atomicAdd(&s_cnt[1], npre);
  }
  __syncthreads();
  int n_mand = s_cnt[0];
  if (threadIdx.x == 0) { w.hd[h].n_mand = n_mand; w.hd[h].n_pre = s_cnt[1]; }
  if (e == 0) return;
  if (n_mand > e) {   // the prefix was feasible, so this cannot happen
    if (threadIdx.x == 0) dev_fail(w.L, DEV_INCONSISTENT, 2000 + h);
    return;
  }
  // Eviction policy: threshold crossers first (default and mandatory + source), or none
  // (densest-only); the rest by decreasing rho~(r) or, for mandatory + source, in
  // provenance order: every key ties, so the provenance selection below takes the oldest.
  const bool mand_first = eviction != DKV_EVICT_DENSEST;
  const bool by_source = eviction == DKV_EVICT_MANDATORY_SOURCE;
  if (!mand_first) n_mand = 0;
  const int k = e - n_mand;   // states to evict after the mandatory ones
  auto is_mand = [&](int i) -> bool {
    if (!mand_first) return false;
    return staged ? ((smand[i >> 5] >> (i & 31)) & 1u) != 0u : (r > 0 && cross[i] <= r);
  };
  auto key_of = [&](int i) -> unsigned { return by_source ? 0u : (staged ? skey[i] : fkey(rt[i])); };
  // radix select of the k-th largest key among non-mandatory states
  unsigned prefix = 0, mask = 0;
  if (threadIdx.x == 0) { s_prefix = 0; s_kk = (unsigned)k; }
  __syncthreads();
  if (k > 0) {
    for (int shift = 24; shift >= 0; shift -= 8) {
      for (int i = threadIdx.x; i < 256; i += blockDim.x) s_hist[i] = 0;
      __syncthreads();
      for (int base = 0; base < m; base += blockDim.x) {
        const int i = base + threadIdx.x;
        bool v = false;
        unsigned key = 0;
        if (i < m && !is_mand(i)) {
          key = key_of(i);
          v = (key & mask) == prefix;
        }
        hist_add(s_hist, v, (key >> shift) & 255u);
      }
      __syncthreads();
      if (warp_id() == 0) {
        unsigned bin, rest;
        if (find_bin(s_hist, s_kk, true, &bin, &rest)) {
          if (lane_id() == 0) { s_kk = rest; s_prefix = prefix | (bin << shift); }
        } else if (lane_id() == 0) {
          dev_fail(w.L, DEV_INCONSISTENT, 2100 + h);
        }
      }
      __syncthreads();
      prefix = s_prefix;
      mask |= 255u << shift;
    }
  }
  const unsigned T = prefix;          // key of the k-th largest
  const unsigned take_eq = s_kk;      // how many states with key == T to evict
  // ties at the threshold: evict the older states (smaller (step, src)) first
  int n_eq_local = 0;
  if (k > 0)
    for (int i = threadIdx.x; i < m; i += blockDim.x)
      if (!is_mand(i) && key_of(i) == T) ++n_eq_local;
  __syncthreads();
  if (threadIdx.x == 0) s_cnt[0] = 0;
  __syncthreads();
  n_eq_local = __reduce_add_sync(0xffffffffu, n_eq_local);
  if (lane_id() == 0) atomicAdd(&s_cnt[0], n_eq_local);
  __syncthreads();
  const unsigned n_eq = (unsigned)s_cnt[0];
  unsigned long long tprefix = 0, tmask = 0;
  const bool need_tie = k > 0 && n_eq > take_eq;
  if (need_tie) {
    if (threadIdx.x == 0) { s_tprefix = 0; s_kk = take_eq; }
    __syncthreads();
    for (int shift = 56; shift >= 0; shift -= 8) {
      for (int i = threadIdx.x; i < 256; i += blockDim.x) s_hist[i] = 0;
      __syncthreads();
      for (int base = 0; base < m; base += blockDim.x) {
        const int i = base + threadIdx.x;
        bool v = false;
        unsigned long long tk = 0;
        if (i < m && !is_mand(i) && key_of(i) == T) {
          tk = ((unsigned long long)(uint32_t)b.prov_step[bh + i] << 32) | (uint32_t)b.prov_src[bh + i];
          v = (tk & tmask) == tprefix;
        }
        hist_add(s_hist, v, (unsigned)((tk >> shift) & 255ull));
      }
      __syncthreads();
      if (warp_id() == 0) {   // smallest first
        unsigned bin, rest;
        if (find_bin(s_hist, s_kk, false, &bin, &rest)) {
          if (lane_id() == 0) { s_kk = rest; s_tprefix = tprefix | ((unsigned long long)bin << shift); }
        } else if (lane_id() == 0) {
          dev_fail(w.L, DEV_INCONSISTENT, 2200 + h);
        }
      }
      __syncthreads();
      tprefix = s_tprefix;
      tmask |= 255ull << shift;
    }
  }
  // provenance keys are unique per head, so "<= tprefix" selects exactly take_eq states
  int n_ev = 0, n_sv = 0;
  for (int base = 0; base < m; base += blockDim.x) {
    const int i = base + threadIdx.x;
    int ev = 0;
    if (i < m) {
      const bool mand = is_mand(i);
      if (mand) ev = 1;
      else if (k > 0) {
        const unsigned key = key_of(i);
        if (key > T) ev = 1;
        else if (key == T) {
          if (!need_tie) ev = 1;
          else {
            const unsigned long long tk = ((unsigned long long)(uint32_t)b.prov_step[bh + i] << 32) |
                                          (uint32_t)b.prov_src[bh + i];
            ev = tk <= tprefix;
          }
        }
      }
    }
    int tot;
    const int off = block_scan_flag(ev, s_warp, &tot);
    if (i < m && ev && n_ev + off < e) w.evict_list[(int64_t)h * b.n_max + n_ev + off] = i;
    const int offs = (threadIdx.x - off);   // survivors before this thread in the chunk
    if (i < m && !ev && n_sv + offs < m) w.surv_list[bh + n_sv + offs] = i;
    n_ev += tot;
    n_sv += min((int)blockDim.x, m - base) - tot;
  }
  if (threadIdx.x == 0 && n_ev != e) dev_fail(w.L, DEV_INCONSISTENT, 3000 + h);
}

// 1 / b of every occupied bank slot (after an import; the update keeps it in step).
__global__ void k_inv_base(Bank b, Ws w) {
  const int h = blockIdx.y;
  const int m = min(max(b.occ[h], 0), b.M_max);
  for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < m; i += gridDim.x * blockDim.x)
    w.invb[(int64_t)h * w.invb_stride + i] = __frcp_rn(b.base[(int64_t)h * b.M_max + i]);
}

// Eq. 12 and the copies Eq. C.4 needs, in one pass.  Rows [0, ns) (only if e > 0): the
// surviving states' keys are copied to the workspace (rows of the subtraction).  Then j:
// for j < e the evicted slot's old key is copied out (columns of the subtraction) and,
// by the same thread, the j-th admitted candidate (pi order) is written over it; the
// admitted candidates j >= e are appended after the old occupancy.  Keys and values
// are copied bit for bit.  An evicted slot is read and overwritten by one thread in
// program order, appended slots lie above every survivor, so no slot is written while
// another thread still reads it.
__global__ void k_commit(Bank b, Ws w, const char* __restrict__ Vc, int N, int esize,
                         const int32_t* __restrict__ src_map) {
  const int h = blockIdx.y;
  const DevHead hd = w.hd[h];
  const int64_t bh = (int64_t)h * b.M_max;
  const int64_t hn = (int64_t)h * b.n_max;
  const int ns = hd.m_old - hd.e;
  if (blockIdx.x == 0 && threadIdx.x == 0) {
    const int m_new = ns + hd.r;
    w.hd[h].m_new = m_new;
    b.occ[h] = m_new;
    if (m_new > hd.M || hd.e > hd.r) dev_fail(w.L, DEV_INCONSISTENT, 4000 + h);
  }
  const int rb = b.d * esize;
  const int kg = rb / 64;          // per row: key groups, value groups, one extension group
  const int per_row = 2 * kg + 1;
  // survivors are operands of the subtraction only when something is evicted (select
  // lists them only then)
  const int ng = hd.e > 0 ? ns : 0;
  const int total = (ng + hd.r) * per_row;
  for (int c = blockIdx.x * blockDim.x + threadIdx.x; c < total; c += gridDim.x * blockDim.x) {
    const int row = c / per_row, grp = c - row * per_row;
    if (row < ng) {
      // surviving state: key and its derived rows to the workspace (its value too with
      // the [K; V] descriptor)
      const int slot = w.surv_list[bh + row];
      if (slot < 0 || slot >= hd.m_old) {
        if (grp == 0) dev_fail(w.L, DEV_INCONSISTENT, 7000 + h);
        continue;
      }
      if (grp < kg) {
        copy64(reinterpret_cast<const uint4*>((const char*)b.k + (bh + slot) * rb) + 4 * grp,
               reinterpret_cast<uint4*>((char*)w.ksurv + (bh + row) * rb) + 4 * grp);
      } else if (grp < 2 * kg) {
        if (w.vsurv)   // [K; V] descriptor: the survivors' values too
          copy64(reinterpret_cast<const uint4*>((const char*)b.v + (bh + slot) * rb) + 4 * (grp - kg),
                 reinterpret_cast<uint4*>((char*)w.vsurv + (bh + row) * rb) + 4 * (grp - kg));
      } else {
        w.ksurv_norm[bh + row] = b.knorm[bh + slot];
        copy64(reinterpret_cast<const uint4*>((const char*)w.bext + (bh + slot) * 64),
               reinterpret_cast<uint4*>((char*)w.ksurv_ext + (bh + row) * 64));
      }
      continue;
    }
    const int j = row - ng;
    const int slot = j < hd.e ? w.evict_list[hn + j] : hd.m_old + (j - hd.e);
    const int src = w.perm[hn + j];
    if (slot < 0 || slot >= hd.M || (j < hd.e && slot >= hd.m_old) || src < 0 || src >= N) {
      if (grp == 0) dev_fail(w.L, DEV_INCONSISTENT, 5000 + h);
      continue;
    }
    if (grp < kg) {
      uint4* dst = reinterpret_cast<uint4*>((char*)b.k + (bh + slot) * rb) + 4 * grp;
      if (j < hd.e) copy64(dst, reinterpret_cast<uint4*>((char*)w.kevict + (hn + j) * rb) + 4 * grp);
      copy64(reinterpret_cast<const uint4*>((const char*)w.kperm + (hn + j) * rb) + 4 * grp, dst);
    } else if (grp < 2 * kg) {
      uint4* dst = reinterpret_cast<uint4*>((char*)b.v + (bh + slot) * rb) + 4 * (grp - kg);
      if (w.vevict && j < hd.e) copy64(dst, reinterpret_cast<uint4*>((char*)w.vevict + (hn + j) * rb) + 4 * (grp - kg));
      copy64(reinterpret_cast<const uint4*>(Vc + ((int64_t)h * N + src) * rb) + 4 * (grp - kg), dst);
    } else {
      uint4* dx = reinterpret_cast<uint4*>((char*)w.bext + (bh + slot) * 64);
      if (j < hd.e) {
        w.kevict_norm[hn + j] = b.knorm[bh + slot];
        copy64(dx, reinterpret_cast<uint4*>((char*)w.kevict_ext + (hn + j) * 64));
      }
      b.knorm[bh + slot] = w.kperm_norm[hn + j];
      b.prov_step[bh + slot] = layer_of(w, h)->step;
      b.prov_src[bh + slot] = src_map ? src_map[(int64_t)h * N + src] : src;
      w.slot_new[hn + j] = slot;
      copy64(reinterpret_cast<const uint4*>((const char*)w.kperm_ext + (hn + j) * 64), dx);
    }
  }
}

// The block's keys, values and source indices in pi order (sequential admission:
// position j of every head is offered together).  Rows are copied bit for bit.
__global__ void k_seq_gather(Bank b, Ws w, const char* __restrict__ Kc, const char* __restrict__ Vc, int N,
                             int esize, char* __restrict__ Kseq, char* __restrict__ Vseq, int32_t* __restrict__ srcseq) {
  const int h = blockIdx.y;
  const int rb = b.d * esize;
  const int kg = rb / 64;   // per position: key groups, value groups
  const int64_t hn = (int64_t)h * b.n_max;
  for (int c = blockIdx.x * blockDim.x + threadIdx.x; c < N * 2 * kg; c += gridDim.x * blockDim.x) {
    const int j = c / (2 * kg), grp = c - j * (2 * kg);
    const int src = w.perm[hn + j];
    if (src < 0 || src >= N) {
      if (grp == 0) dev_fail(w.L, DEV_INCONSISTENT, 8600 + h);
      continue;
    }
    const int64_t so = ((int64_t)h * N + src) * rb, dof = ((int64_t)h * N + j) * rb;
    if (grp < kg) copy64(reinterpret_cast<const uint4*>(Kc + so) + 4 * grp, reinterpret_cast<uint4*>(Kseq + dof) + 4 * grp);
    else copy64(reinterpret_cast<const uint4*>(Vc + so) + 4 * (grp - kg), reinterpret_cast<uint4*>(Vseq + dof) + 4 * (grp - kg));
    if (grp == 0) srcseq[(int64_t)h * N + j] = src;
  }
}

}  // namespace

static float ext_goff(const KParams& kp) { return kp.eps * 0.5f / kp.inv_s2; }   // eps sigma^2 / 2

cudaError_t launch_cand_norms(const Bank& b, const Ws& w, const void* Kc, const void* Vc, int N, int64_t step,
                              const KParams& kp, const RopeArgs* rope, cudaStream_t s, Timer* t) {
  if (!w.vperm) Vc = nullptr;   // values enter the norms with the [K; V] descriptor only
  dim3 grid((N + 8 * NR_ROWS - 1) / (8 * NR_ROWS) + 1, b.H);   // + the prepare block
  timer_begin(t, "cand_norms", s);
  if (rope) {
    const dim3 rgrid((N + ROPE_ROWS - 1) / ROPE_ROWS + 1);   // + the prepare block
    if (b.bf16)
      k_cand_prepare_rope<__nv_bfloat16><<<rgrid, 256, 0, s>>>(b, w, (const __nv_bfloat16*)Kc,
                                                               (const __nv_bfloat16*)Vc, N, step, ext_goff(kp), *rope);
    else
      k_cand_prepare_rope<float><<<rgrid, 256, 0, s>>>(b, w, (const float*)Kc, (const float*)Vc, N, step,
                                                       ext_goff(kp), *rope);
  } else if (b.bf16) {
    k_cand_prepare<__nv_bfloat16><<<grid, 256, 0, s>>>(b, w, (const __nv_bfloat16*)Kc, (const __nv_bfloat16*)Vc, N,
                                                       step, ext_goff(kp));
  } else {
    k_cand_prepare<float><<<grid, 256, 0, s>>>(b, w, (const float*)Kc, (const float*)Vc, N, step, ext_goff(kp));
  }
  timer_end(t, s);
  return cudaGetLastError();
}

cudaError_t launch_bank_norms(const Bank& b, const Ws& w, const KParams& kp, cudaStream_t s, Timer* t) {
  dim3 grid((b.M_max + 8 * NR_ROWS - 1) / (8 * NR_ROWS), b.H);
  __nv_bfloat16* ext = (__nv_bfloat16*)w.bext;
  timer_begin(t, "bank_norms", s);
  const void* V = w.vperm ? b.v : nullptr;   // [K; V] descriptor: norms of [k; v]
  if (b.bf16)
    k_row_norms<__nv_bfloat16><<<grid, 256, 0, s>>>((const __nv_bfloat16*)b.k, (const __nv_bfloat16*)V,
                                                    (int64_t)b.M_max * b.d, b.M_max, b.occ, 1, 0, b.knorm, b.M_max,
                                                    b.d, ext, (int64_t)b.M_max * 32, ext_goff(kp));
  else
    k_row_norms<float><<<grid, 256, 0, s>>>((const float*)b.k, (const float*)V, (int64_t)b.M_max * b.d, b.M_max,
                                            b.occ, 1, 0, b.knorm, b.M_max, b.d, ext, (int64_t)b.M_max * 32,
                                            ext_goff(kp));
  timer_end(t, s);
  return cudaGetLastError();
}

cudaError_t launch_inv_base(const Bank& b, const Ws& w, cudaStream_t s) {
  dim3 grid((b.M_max + 255) / 256, b.H);
  k_inv_base<<<grid, 256, 0, s>>>(b, w);
  return cudaGetLastError();
}

cudaError_t launch_sort(const Bank& b, const Ws& w, const void* Kc, const void* Vc, int identity, cudaStream_t s,
                        Timer* t) {
  const int max_runs = (b.n_max + RUN - 1) / RUN;
  timer_begin(t, "sort_runs", s);
  k_sort_runs<<<dim3((max_runs + 7) / 8, b.H), 256, 0, s>>>(w, b.n_max, identity);
  timer_end(t, s);
  timer_begin(t, "sort_rank", s);
  // four runs per CTA (1,024 threads) when that still gives every SM two CTAs: each CTA
  // loads every run of its head into shared memory once for four runs (config 4: 1.35 ms
  // with one run per CTA, 1.16 with two, 1.13 with four); one run per CTA otherwise (config
  // 1, 228 runs: 22 us against 33 with four)
  const int n_sm = sm_count();
  const size_t sm_bytes = (size_t)max_runs * RUN * 8;
  if ((int64_t)b.H * ((max_runs + 3) / 4) >= 2 * (int64_t)n_sm)
    k_sort_rank<4><<<dim3((max_runs + 3) / 4, b.H), RUN * 4, sm_bytes, s>>>(b, w, (const char*)Kc, (const char*)Vc,
                                                                          b.bf16 ? 2 : 4, identity);
  else
    k_sort_rank<1><<<dim3(max_runs, b.H), RUN, sm_bytes, s>>>(b, w, (const char*)Kc, (const char*)Vc,
                                                             b.bf16 ? 2 : 4, identity);
  timer_end(t, s);
  return cudaGetLastError();
}

cudaError_t launch_rstar(const Bank& b, const Ws& w, const KParams& kp, cudaStream_t s, Timer* t) {
  timer_begin(t, "rstar", s);
  k_rstar<<<b.H, BIG, 0, s>>>(b, w, kp.sync_heads);
  timer_end(t, s);
  return cudaGetLastError();
}

cudaError_t launch_select(const Bank& b, const Ws& w, int eviction, cudaStream_t s, Timer* t) {
  timer_begin(t, "select", s);
  k_select<<<b.H, BIG, sel_smem_bytes(b.M_max), s>>>(b, w, eviction);
  timer_end(t, s);
  return cudaGetLastError();
}

cudaError_t launch_commit(const Bank& b, const Ws& w, const void* Vc, int N, const int32_t* src_map, cudaStream_t s,
                          Timer* t) {
  // rows: ns survivors + r admitted = m_new <= M_max per head, grid-stride over them.  A
  // head's CTAs cover its largest possible row range in one pass only when the heads are
  // few: with many heads, whose layers mostly admit nothing, each head gets a few CTAs
  // (a grid sized for the largest budget spent 0.6 ms per step starting empty CTAs at
  // 1,600 heads)
  const int full = (b.M_max * (2 * b.d * (b.bf16 ? 2 : 4) / 64 + 1) + 255) / 256;
  const int n_sm = sm_count();
  const int want = n_sm > 0 ? std::max(2, (16 * n_sm + b.H - 1) / b.H) : full;
  dim3 grid(std::min(full, want), b.H);
  timer_begin(t, "commit", s);
  k_commit<<<grid, 256, 0, s>>>(b, w, (const char*)Vc, N, b.bf16 ? 2 : 4, src_map);
  timer_end(t, s);
  return cudaGetLastError();
}

cudaError_t launch_seq_gather(const Bank& b, const Ws& w, const void* Kc, const void* Vc, int N, void* Kseq,
                              void* Vseq, int32_t* srcseq, cudaStream_t s) {
  const int kg = b.d * (b.bf16 ? 2 : 4) / 64;
  dim3 grid((N * 2 * kg + 255) / 256, b.H);
  k_seq_gather<<<grid, 256, 0, s>>>(b, w, (const char*)Kc, (const char*)Vc, N, b.bf16 ? 2 : 4, (char*)Kseq,
                                    (char*)Vseq, srcseq);
  return cudaGetLastError();
}

cudaError_t update_set_smem_limits() {
  // phase 2 of the sort holds every run of a head: up to 64 runs of 2 KiB
  cudaError_t e = cudaFuncSetAttribute(k_sort_rank<1>, cudaFuncAttributeMaxDynamicSharedMemorySize, 64 * RUN * 8);
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(k_sort_rank<4>, cudaFuncAttributeMaxDynamicSharedMemorySize, 64 * RUN * 8);
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(k_select, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sel_smem_bytes(SEL_STAGE));
  return e;
}

}  // namespace dkv
