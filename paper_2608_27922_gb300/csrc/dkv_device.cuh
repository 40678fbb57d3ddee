// Device-side shared definitions of the DensityKV GB300 library.
//
// Layouts (all row-major, innermost d):
//   bank k / v        [H][M_max][d]   (caller-owned)
//   rho, base, knorm  [H][M_max] fp32 (caller-owned)
//   candidates        [H][N][d]       (caller-owned, valid from admit to compress)
//   workspace         carved by dkv_api.cu (see WsLayout there)
#pragma once

#include <cuda_runtime.h>
#include <cuda_bf16.h>
#include <stdint.h>

namespace dkv {

// Device error word codes (mirrors dkv_status_t values for the sticky errors).
enum : int32_t { DEV_OK = 0, DEV_TIMEOUT = 6, DEV_INCONSISTENT = 8 };

// Per-layer device state, written by the update kernels.
struct DevLayer {
  int32_t N;           // candidates of the current update
  int32_t rmax;        // min(N, min over live heads of M_h)
  int32_t r_star;      // shared prefix (max over heads when heads are independent)
  int32_t empty_all;   // every head took the empty-bank path
  int64_t step;        // provenance step of the current update
  int32_t err;         // sticky error word (DEV_*)
  int32_t err_info;    // first failing site (kernel-specific code)
  int32_t arrive;      // arrival counter of the r* kernel's head blocks (0 between launches)
};

// Per-head device state.
struct DevHead {
  int32_t m_old;     // occupancy when admit ran
  int32_t M;         // budget M_h
  int32_t r;         // candidates admitted in this head (r* or r*_h, or min(N, M_h) if empty)
  int32_t e;         // evictions e_{r} = max(0, m_old + r - M)
  int32_t n_mand;    // mandatory evictions
  int32_t n_pre;     // pre-violators (g(0) >= tau)
  int32_t m_new;     // occupancy after commit
  int32_t empty;     // 1 if the head took the empty-bank path
};

// Soft-Riesz parameters in the form the kernels use (Eq. 2).
struct KParams {
  float inv_s2;      // 1 / sigma^2
  float eps;
  float tau;
  float delta;
  int32_t p;         // 1, 2 or 4
  int32_t sync_heads;
  int32_t order;     // dkv_order_t
  int32_t eviction;  // dkv_evict_t
  int32_t refresh;   // 1: b = max(rho, delta) for every retained state after each update
};

// Snapshots of the running prefix sum of Eq. C.2 are kept every SNAP columns.
constexpr int SNAP = 128;

template <typename T> __device__ __forceinline__ float to_f(T x);
template <> __device__ __forceinline__ float to_f<float>(float x) { return x; }
template <> __device__ __forceinline__ float to_f<__nv_bfloat16>(__nv_bfloat16 x) { return __bfloat162float(x); }

// w = (eps + d2 / sigma^2)^(-p) for integer p in {1, 2, 4}, with IEEE-rounded
// operations so that every kernel that evaluates a pair gets the same bits.
__device__ __forceinline__ float riesz_w(float d2, const KParams& kp) {
  float u = __fmaf_rn(d2, kp.inv_s2, kp.eps);
  float r = __frcp_rn(u);
  if (kp.p == 1) return r;
  float r2 = __fmul_rn(r, r);
  if (kp.p == 2) return r2;
  return __fmul_rn(r2, r2);
}

// Records the first device-side failure in the layer's sticky error word.
__device__ __forceinline__ void dev_fail(DevLayer* L, int32_t code, int32_t info) {
  if (atomicCAS(&L->err, 0, code) == 0) atomicExch(&L->err_info, info);
}

__device__ __forceinline__ uint64_t globaltimer_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

// Monotone map of floats to unsigned keys (a < b  =>  fkey(a) < fkey(b); -0 below +0).
__device__ __forceinline__ uint32_t fkey(float x) {
  uint32_t u = __float_as_uint(x);
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

}  // namespace dkv
