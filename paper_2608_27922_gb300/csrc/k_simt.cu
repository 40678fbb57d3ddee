// fp32 "exactness mode" kernels: every candidate/bank interaction is evaluated
// on the CUDA cores as a direct sum of squared differences,
//   d2 = sum_k (a_k - b_k)^2   (fp32, sequential fused multiply-adds),
// then w = (eps + d2 / sigma^2)^(-p) (Eq. 2).  These kernels serve fp32 banks
// and the DKV_SCORE_FP32 mode of bf16 banks.
//
// Two neighbouring threads share two rows: each holds one half of the dimensions of
// both rows, forms the two half sums (sequential fused multiply-adds), and one shuffle
// gives each thread d2 = first half + second half of its own row (same order in every
// pass).  Each thread walks the columns in increasing order, so the running sums of
// Eq. C.2 are formed in the same order by the crossing pass and by the projection pass
// that later resumes them from a snapshot.  Every staged column element thus serves
// two rows (half the shared-memory reads of a one-row-per-thread layout).
// With the [K; V] descriptor (App. E "Retention geometry") two neighbouring threads
// own one row, one its key and one its value; d2 = d2_key + d2_value after one shuffle,
// identical in both, and the even thread writes.
#include "dkv_internal.h"

#include <climits>

namespace dkv {

namespace {

enum PMode { PM_SCORE = 0, PM_CROSS = 1, PM_PROJECT = 2, PM_SUB = 3, PM_NEWBASE = 4 };

constexpr int ROWS = 128;   // rows (threads) per block
constexpr int CT = 32;      // columns staged per shared-memory tile

struct PairJob {
  const void* rk;    // row keys of head 0
  int64_t rk_hs;     // row-key head stride (elements)
  const void* ck;    // column keys of head 0
  int64_t ck_hs;     // column-key head stride (elements)
  const void* rv;    // row values ([K; V] descriptor; same layout as rk)
  const void* cv;    // column values (same layout as ck)
  Bank b;
  Ws w;
  KParams kp;
};

template <typename T>
__device__ __forceinline__ const T* ptr(const void* p, int64_t off) {
  return reinterpret_cast<const T*>(p) + off;
}

template <typename T, int D, int MODE, bool KV>
__global__ void __launch_bounds__(ROWS) simt_pairs(PairJob j) {
  constexpr int DC = KV ? 2 * D : D;   // staged floats per column: key (| value)
  constexpr int RPB = KV ? ROWS / 2 : ROWS;   // rows per block
  constexpr int DH = D / 2;
  extern __shared__ float smem[];
  float* cs = smem;               // [CT][DC] staged column keys (| values)
  float* cmeta = smem + CT * DC;  // [CT]     per-column factor (SCORE: 1 / b_j)

  const int h = blockIdx.y;
  const DevHead hd = j.w.hd[h];
  const int N = layer_of(j.w, h)->N;
  const int rmax = layer_of(j.w, h)->rmax;
  int nrows = 0, c0 = 0, c1 = 0;
  if (MODE == PM_SCORE) { nrows = hd.empty ? 0 : N;                 c1 = hd.m_old; }
  if (MODE == PM_CROSS) { nrows = hd.empty ? 0 : hd.m_old;          c1 = rmax; }
  if (MODE == PM_PROJECT) { nrows = hd.empty ? 0 : hd.m_old;        c0 = (hd.r / SNAP) * SNAP; c1 = hd.r; }
  if (MODE == PM_SUB) { nrows = hd.empty ? 0 : hd.m_old - hd.e;     c1 = hd.e; }
  if (MODE == PM_NEWBASE) { nrows = hd.r;                           c1 = hd.m_new; }
  const int row0 = blockIdx.x * RPB;
  if (row0 >= nrows) return;
  const int half = threadIdx.x & 1;   // KV: 0 key, 1 value; else: dimensions [half D/2, +D/2)
  const int pr = threadIdx.x >> 1;
  const int row = KV ? row0 + pr : row0 + 2 * pr + half;
  const bool active = row < nrows;
  const bool writer = KV ? active && half == 0 : active;
  const int64_t bh = (int64_t)h * j.b.M_max;   // bank head offset (rows)

  // KV: this thread's row key (or value); else halves of the pair's two rows:
  // rr[0, D/2) = row 2 pr, rr[D/2, D) = row 2 pr + 1, dimensions [half D/2, half D/2 + D/2)
  float rr[D];
  if (KV) {
    const T* rp = ptr<T>(half ? j.rv : j.rk, (int64_t)h * j.rk_hs + (int64_t)(active ? row : 0) * D);
#pragma unroll
    for (int k = 0; k < D; ++k) rr[k] = active ? to_f<T>(rp[k]) : 0.f;
  } else {
#pragma unroll
    for (int q = 0; q < 2; ++q) {
      const int rq = row0 + 2 * pr + q;
      const bool aq = rq < nrows;
      const T* rp = ptr<T>(j.rk, (int64_t)h * j.rk_hs + (int64_t)(aq ? rq : 0) * D + half * DH);
#pragma unroll
      for (int k = 0; k < DH; ++k) rr[q * DH + k] = aq ? to_f<T>(rp[k]) : 0.f;
    }
  }

  // per-row state
  float S = 0.f, acc = 0.f, thr = 0.f;
  int cross = INT_MAX, self = -1, slot = -1;
  float* snap_row = nullptr;
  if (active) {
    if (MODE == PM_CROSS) {
      S = j.b.rho[bh + row];
      thr = __fmul_rn(j.kp.tau, j.b.base[bh + row]);
      if (S >= thr) cross = 0;
      snap_row = j.w.snap + ((int64_t)h * j.b.M_max + row) * j.w.snap_stride;
      if (writer) snap_row[0] = S;
    } else if (MODE == PM_PROJECT) {
      S = j.w.snap[((int64_t)h * j.b.M_max + row) * j.w.snap_stride + c0 / SNAP];
    } else if (MODE == PM_SUB) {
      // with no eviction every state survives in place and rho := rho~(r) (Eq. C.4)
      slot = hd.e == 0 ? row : j.w.surv_list[(int64_t)h * j.b.M_max + row];
    } else if (MODE == PM_NEWBASE) {
      self = j.w.slot_new[(int64_t)h * j.b.n_max + row];
    }
  }

  for (int t0 = c0; t0 < c1; t0 += CT) {
    const int nc = min(CT, c1 - t0);
    __syncthreads();
    const T* cp = ptr<T>(j.ck, (int64_t)h * j.ck_hs + (int64_t)t0 * D);
    if (KV) {
      const T* cvp = ptr<T>(j.cv, (int64_t)h * j.ck_hs + (int64_t)t0 * D);
      for (int e = threadIdx.x; e < nc * DC; e += ROWS) {
        const int c = e / DC, k = e - c * DC;
        cs[e] = to_f<T>(k < D ? cp[c * D + k] : cvp[c * D + k - D]);
      }
    } else {
      for (int e = threadIdx.x; e < nc * D; e += ROWS) cs[e] = to_f<T>(cp[e]);
    }
    if (MODE == PM_SCORE)
      for (int c = threadIdx.x; c < nc; c += ROWS) cmeta[c] = __frcp_rn(j.b.base[bh + t0 + c]);
    __syncthreads();
    // every thread takes part in the shuffles (a thread whose row is past the end too)
    for (int c = 0; c < nc; ++c) {
      float d2;
      if (KV) {
        const float* col = cs + c * DC + half * D;
        d2 = 0.f;
#pragma unroll
        for (int k = 0; k < D; ++k) {
          float df = __fsub_rn(rr[k], col[k]);
          d2 = __fmaf_rn(df, df, d2);
        }
        const float other = __shfl_xor_sync(0xffffffffu, d2, 1);
        d2 = half ? __fadd_rn(other, d2) : __fadd_rn(d2, other);   // key part + value part
      } else {
        const float* col = cs + c * DC + half * DH;
        float q0 = 0.f, q1 = 0.f;
#pragma unroll
        for (int k = 0; k < DH; ++k) {
          const float x = col[k];
          const float d0 = __fsub_rn(rr[k], x), d1 = __fsub_rn(rr[DH + k], x);
          q0 = __fmaf_rn(d0, d0, q0);
          q1 = __fmaf_rn(d1, d1, q1);
        }
        // the partner needs this thread's half of its row: row 2 pr + 1 - half
        const float other = __shfl_xor_sync(0xffffffffu, half ? q0 : q1, 1);
        d2 = half ? __fadd_rn(other, q1) : __fadd_rn(q0, other);    // first half + second half
      }
      const float w = riesz_w(d2, j.kp);
      const int jc = t0 + c;
      if (MODE == PM_SCORE) {
        acc = __fmaf_rn(w, cmeta[c], acc);
      } else if (MODE == PM_CROSS) {
        S = __fadd_rn(S, w);
        if (cross == INT_MAX && S >= thr) cross = jc + 1;
        if (writer && ((jc + 1) % SNAP) == 0) snap_row[(jc + 1) / SNAP] = S;
      } else if (MODE == PM_PROJECT) {
        S = __fadd_rn(S, w);
      } else if (MODE == PM_SUB) {
        acc = __fadd_rn(acc, w);
      } else {
        if (jc != self) S = __fadd_rn(S, w);
      }
    }
  }
  if (!writer) return;
  if ((MODE == PM_SUB && (slot < 0 || slot >= hd.m_old)) || (MODE == PM_NEWBASE && (self < 0 || self >= hd.M))) {
    dev_fail(j.w.L, DEV_INCONSISTENT, 6000 + MODE);   // a list entry out of range: skip the write
    return;
  }
  if (MODE == PM_SCORE) {
    j.w.score[(int64_t)h * j.b.n_max + row] = __fdiv_rn(acc, (float)hd.m_old);
  } else if (MODE == PM_CROSS) {
    j.w.cross[bh + row] = cross;
    const int bin = cross == INT_MAX ? rmax + 1 : cross;
    atomicAdd(&j.w.hist[(int64_t)h * j.w.hist_stride + bin], 1);
  } else if (MODE == PM_PROJECT) {
    j.w.rho_t[bh + row] = S;
  } else if (MODE == PM_SUB) {
    const float rho = __fsub_rn(j.w.rho_t[bh + slot], acc);
    j.b.rho[bh + slot] = rho;
    if (j.kp.refresh) {   // refreshed-baseline policy: b follows the current density
      const float bnew = fmaxf(rho, j.kp.delta);
      j.b.base[bh + slot] = bnew;
      j.w.invb[(int64_t)h * j.w.invb_stride + slot] = __frcp_rn(bnew);
    }
  } else {
    j.b.rho[bh + self] = S;
    const float bnew = fmaxf(S, j.kp.delta);
    j.b.base[bh + self] = bnew;
    j.w.invb[(int64_t)h * j.w.invb_stride + self] = __frcp_rn(bnew);
  }
}

template <int MODE, bool KV>
void launch_pairs_t(dim3 grid, size_t sm, cudaStream_t s, const Bank& b, const PairJob& j) {
  if (b.bf16) {
    if (b.d == 128) simt_pairs<__nv_bfloat16, 128, MODE, KV><<<grid, ROWS, sm, s>>>(j);
    else simt_pairs<__nv_bfloat16, 64, MODE, KV><<<grid, ROWS, sm, s>>>(j);
  } else {
    if (b.d == 128) simt_pairs<float, 128, MODE, KV><<<grid, ROWS, sm, s>>>(j);
    else simt_pairs<float, 64, MODE, KV><<<grid, ROWS, sm, s>>>(j);
  }
}

// rv / cv: the row and column values, non-null only with the [K; V] descriptor.
template <int MODE>
cudaError_t launch_pairs(const Bank& b, const Ws& w, const KParams& kp, const void* rk, int64_t rk_hs,
                         const void* ck, int64_t ck_hs, const void* rv, const void* cv, int max_rows,
                         cudaStream_t s, Timer* t, const char* name) {
  const bool kv = rv != nullptr;
  PairJob j{rk, rk_hs, ck, ck_hs, rv, cv, b, w, kp};
  const int rpb = kv ? ROWS / 2 : ROWS;
  dim3 grid((max_rows + rpb - 1) / rpb, b.H);
  if (grid.x == 0) return cudaSuccess;
  const size_t sm = (size_t)(CT * b.d * (kv ? 2 : 1) + CT) * sizeof(float);
  timer_begin(t, name, s);
  if (kv) launch_pairs_t<MODE, true>(grid, sm, s, b, j);
  else launch_pairs_t<MODE, false>(grid, sm, s, b, j);
  timer_end(t, s);
  return cudaGetLastError();
}

// ---------------------------------------------------------------- attention
constexpr int AQ = 128;   // queries per block
constexpr int AK = 32;    // keys per shared-memory tile

template <typename T, int D>
__global__ void __launch_bounds__(AQ) simt_attend(const T* __restrict__ Q, int Nq, const T* __restrict__ Kw,
                                                  const T* __restrict__ Vw, int W, T* __restrict__ O, Bank b,
                                                  float qscale) {
  extern __shared__ float smem[];
  float* qs = smem;                 // [D][AQ] queries, transposed
  float* ks = qs + D * AQ;          // [AK][D]
  float* vs = ks + AK * D;          // [AK][D]
  const int h = blockIdx.y;
  const int q0 = blockIdx.x * AQ;
  const int qi = q0 + threadIdx.x;
  const bool active = qi < Nq;
  const int m = min(max(b.occ[h], 0), b.M_max);
  const int nkeys = m + W;
  for (int e = threadIdx.x; e < AQ * D; e += AQ) {
    const int r = e / D, k = e % D;
    const int qq = q0 + r;
    qs[k * AQ + r] = qq < Nq ? to_f<T>(Q[((int64_t)h * Nq + qq) * D + k]) * qscale : 0.f;
  }
  float acc[D];
#pragma unroll
  for (int k = 0; k < D; ++k) acc[k] = 0.f;
  float mrun = -INFINITY, l = 0.f;
  const T* kb = reinterpret_cast<const T*>(b.k) + (int64_t)h * b.M_max * D;
  const T* vb = reinterpret_cast<const T*>(b.v) + (int64_t)h * b.M_max * D;
  const T* kw = Kw + (int64_t)h * W * D;
  const T* vw = Vw + (int64_t)h * W * D;
  for (int t0 = 0; t0 < nkeys; t0 += AK) {
    const int nc = min(AK, nkeys - t0);
    __syncthreads();
    for (int e = threadIdx.x; e < nc * D; e += AQ) {
      const int c = t0 + e / D, k = e % D;
      ks[e] = c < m ? to_f<T>(kb[(int64_t)c * D + k]) : to_f<T>(kw[(int64_t)(c - m) * D + k]);
      vs[e] = c < m ? to_f<T>(vb[(int64_t)c * D + k]) : to_f<T>(vw[(int64_t)(c - m) * D + k]);
    }
    __syncthreads();
    // four keys at a time: each staged query element serves four dot products and the
    // running maximum is raised at most once per four keys
    int c = 0;
#pragma unroll 1
    for (; c + 4 <= nc; c += 4) {
      float a[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll 8
      for (int k = 0; k < D; ++k) {
        const float q = qs[k * AQ + threadIdx.x];
#pragma unroll
        for (int u = 0; u < 4; ++u) a[u] = fmaf(q, ks[(c + u) * D + k], a[u]);
      }
      const float amax = fmaxf(fmaxf(a[0], a[1]), fmaxf(a[2], a[3]));
      if (amax > mrun) {   // online softmax: rescale the running sums to the new maximum
        const float alpha = exp2f(mrun - amax);
        l *= alpha;
#pragma unroll
        for (int k = 0; k < D; ++k) acc[k] *= alpha;
        mrun = amax;
      }
      float pu[4];
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        pu[u] = exp2f(a[u] - mrun);
        l += pu[u];
      }
#pragma unroll
      for (int k = 0; k < D; ++k) {
        float x = acc[k];
#pragma unroll
        for (int u = 0; u < 4; ++u) x = fmaf(pu[u], vs[(c + u) * D + k], x);
        acc[k] = x;
      }
    }
#pragma unroll 1
    for (; c < nc; ++c) {
      float a = 0.f;
#pragma unroll 8
      for (int k = 0; k < D; ++k) a = fmaf(qs[k * AQ + threadIdx.x], ks[c * D + k], a);
      if (a > mrun) {   // online softmax: rescale the running sums to the new maximum
        const float alpha = exp2f(mrun - a);
        l *= alpha;
#pragma unroll
        for (int k = 0; k < D; ++k) acc[k] *= alpha;
        mrun = a;
      }
      const float p = exp2f(a - mrun);
      l += p;
#pragma unroll
      for (int k = 0; k < D; ++k) acc[k] = fmaf(p, vs[c * D + k], acc[k]);
    }
  }
  if (!active) return;
  const float inv = l > 0.f ? 1.f / l : 0.f;
  T* o = O + ((int64_t)h * Nq + qi) * D;
#pragma unroll
  for (int k = 0; k < D; ++k) {
    const float x = acc[k] * inv;
    if constexpr (sizeof(T) == 2) o[k] = __float2bfloat16_rn(x); else o[k] = x;
  }
}

}  // namespace

// With the [K; V] descriptor every pass also reads the values beside its keys: the
// candidates' (source order; pi order: vperm), the bank's, and the survivors' and evicted
// states' copies (vsurv, vevict) taken by commit.
cudaError_t launch_score_fp32(const Bank& b, const Ws& w, const void* Kc, const void* Vc, int N, const KParams& kp,
                              cudaStream_t s, Timer* t) {
  // rows: candidates in source order; columns: bank keys [0, m)
  const bool kv = w.vperm != nullptr;
  return launch_pairs<PM_SCORE>(b, w, kp, Kc, (int64_t)N * b.d, b.k, (int64_t)b.M_max * b.d, kv ? Vc : nullptr,
                                kv ? b.v : nullptr, N, s, t, "score_fp32");
}

cudaError_t launch_cross_fp32(const Bank& b, const Ws& w, const KParams& kp, cudaStream_t s, Timer* t) {
  const bool kv = w.vperm != nullptr;
  return launch_pairs<PM_CROSS>(b, w, kp, b.k, (int64_t)b.M_max * b.d, w.kperm, (int64_t)b.n_max * b.d,
                                kv ? b.v : nullptr, w.vperm, b.M_max, s, t, "cross_fp32");
}

cudaError_t launch_project_fp32(const Bank& b, const Ws& w, const KParams& kp, cudaStream_t s, Timer* t) {
  const bool kv = w.vperm != nullptr;
  return launch_pairs<PM_PROJECT>(b, w, kp, b.k, (int64_t)b.M_max * b.d, w.kperm, (int64_t)b.n_max * b.d,
                                  kv ? b.v : nullptr, w.vperm, b.M_max, s, t, "project_fp32");
}

cudaError_t launch_subtract_fp32(const Bank& b, const Ws& w, const KParams& kp, cudaStream_t s, Timer* t) {
  return launch_pairs<PM_SUB>(b, w, kp, w.ksurv, (int64_t)b.M_max * b.d, w.kevict, (int64_t)b.n_max * b.d,
                              w.vsurv, w.vevict, b.M_max, s, t, "subtract_fp32");
}

cudaError_t launch_newbase_fp32(const Bank& b, const Ws& w, const KParams& kp, cudaStream_t s, Timer* t) {
  const bool kv = w.vperm != nullptr;
  return launch_pairs<PM_NEWBASE>(b, w, kp, w.kperm, (int64_t)b.n_max * b.d, b.k, (int64_t)b.M_max * b.d,
                                  w.vperm, kv ? b.v : nullptr, b.n_max, s, t, "newbase_fp32");
}

cudaError_t launch_attend_fp32(const Bank& b, const void* Q, int Nq, const void* Kw, const void* Vw, int W,
                               void* O, cudaStream_t s, Timer* t) {
  dim3 grid((Nq + AQ - 1) / AQ, b.H);
  const size_t sm = (size_t)(b.d * AQ + 2 * AK * b.d) * sizeof(float);
  const float qscale = 1.4426950408889634f / sqrtf((float)b.d);   // log2(e) / sqrt(d)
  timer_begin(t, "attend_fp32", s);
  if (b.bf16) {
    using T = __nv_bfloat16;
    if (b.d == 128)
      simt_attend<T, 128><<<grid, AQ, sm, s>>>((const T*)Q, Nq, (const T*)Kw, (const T*)Vw, W, (T*)O, b, qscale);
    else
      simt_attend<T, 64><<<grid, AQ, sm, s>>>((const T*)Q, Nq, (const T*)Kw, (const T*)Vw, W, (T*)O, b, qscale);
  } else {
    if (b.d == 128)
      simt_attend<float, 128><<<grid, AQ, sm, s>>>((const float*)Q, Nq, (const float*)Kw, (const float*)Vw, W,
                                                   (float*)O, b, qscale);
    else
      simt_attend<float, 64><<<grid, AQ, sm, s>>>((const float*)Q, Nq, (const float*)Kw, (const float*)Vw, W,
                                                  (float*)O, b, qscale);
  }
  timer_end(t, s);
  return cudaGetLastError();
}

// Dynamic shared memory above 48 KB must be opted into once per kernel.
cudaError_t simt_set_smem_limits() {
  const int a = 227 * 1024;
  cudaError_t e = cudaSuccess;
#define DKV_OPT(K) if (e == cudaSuccess) e = cudaFuncSetAttribute(K, cudaFuncAttributeMaxDynamicSharedMemorySize, a)
  DKV_OPT((simt_attend<float, 128>));
  DKV_OPT((simt_attend<float, 64>));
  DKV_OPT((simt_attend<__nv_bfloat16, 128>));
  DKV_OPT((simt_attend<__nv_bfloat16, 64>));
#undef DKV_OPT
  return e;
}

}  // namespace dkv
