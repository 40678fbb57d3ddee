// dkv_candidate_order_noalloc: candidate scoring and ordering for callers that
// cannot allocate device memory.
//
// The regular path (dkv_bank_admit) keeps its intermediates in a workspace the
// caller allocates.  Some callers cannot allocate at all: code that runs inside a
// framework that owns every device byte through its own pool, real-time or
// embedded hosts where allocation is forbidden after start-up, or plugins that only
// receive pre-sized input and output buffers.  This entry point needs nothing but
// the caller's inputs and outputs: the one scratch buffer it uses (the per-
// candidate scores between the scoring kernel and the ordering kernel) is the
// file-scope device array below, of a fixed size.
//
// The scoring kernel is the fp32 direct-difference variant of the Eq. 6 pass for
// one head, with the arithmetic of the fp32 score mode of dkv_bank_admit in the same
// order: d2 = (sequential fused multiply-adds over the first half of the dimensions)
// + (the same over the second half), one rounded add joining them; w by the shared
// Eq. 2 helper; the weighted sum over bank columns in increasing order; one division
// by m.  Its scores are therefore bit-identical to admit's in that mode.  The ordering
// kernel is the stable ascending sort with ties in source order.
#include "../../include/dkv.h"
#include "dkv_device.cuh"

#include <climits>
#include <cmath>
#include <mutex>

namespace dkv {
namespace {

// Scratch shared by every call on a device, held until the process exits.
static __device__ __align__(256) float g_noalloc_scores[DKV_NOALLOC_MAX_N];

constexpr int ROWS = 128;   // candidates per block of the scoring kernel
constexpr int CT = 32;      // bank keys staged per shared-memory tile
constexpr int SORT_THREADS = 1024;

template <typename T, int D>
__global__ void __launch_bounds__(ROWS) noalloc_score(const T* __restrict__ Kb, const float* __restrict__ base,
                                                      int m, const T* __restrict__ Kc, int N, KParams kp,
                                                      float* __restrict__ scratch) {
  __shared__ float cs[CT * D];
  __shared__ float cinv[CT];
  const int x = blockIdx.x * ROWS + threadIdx.x;
  const bool active = x < N;
  float rr[D];
#pragma unroll
  for (int k = 0; k < D; ++k) rr[k] = active ? to_f<T>(Kc[(int64_t)x * D + k]) : 0.f;
  float acc = 0.f;
  for (int t0 = 0; t0 < m; t0 += CT) {
    const int nc = min(CT, m - t0);
    __syncthreads();
    for (int e = threadIdx.x; e < nc * D; e += ROWS) cs[e] = to_f<T>(Kb[(int64_t)t0 * D + e]);
    for (int c = threadIdx.x; c < nc; c += ROWS) cinv[c] = __frcp_rn(base[t0 + c]);
    __syncthreads();
    if (!active) continue;
    for (int c = 0; c < nc; ++c) {
      const float* col = cs + c * D;
      float q0 = 0.f, q1 = 0.f;   // first and second half of the dimensions
#pragma unroll
      for (int k = 0; k < D / 2; ++k) {
        const float d0 = __fsub_rn(rr[k], col[k]), d1 = __fsub_rn(rr[D / 2 + k], col[D / 2 + k]);
        q0 = __fmaf_rn(d0, d0, q0);
        q1 = __fmaf_rn(d1, d1, q1);
      }
      acc = __fmaf_rn(riesz_w(__fadd_rn(q0, q1), kp), cinv[c], acc);
    }
  }
  if (active) scratch[x] = __fdiv_rn(acc, (float)m);
}

__global__ void __launch_bounds__(SORT_THREADS) noalloc_order(const float* __restrict__ scratch, int N, int m,
                                                              int32_t* __restrict__ perm, float* __restrict__ scores) {
  extern __shared__ unsigned long long keys[];
  if (m == 0) {   // empty bank: source order (Alg. 1, m = 0 branch)
    for (int i = threadIdx.x; i < N; i += blockDim.x) {
      perm[i] = i;
      if (scores) scores[i] = 0.f;
    }
    return;
  }
  int n = 2;
  while (n < N) n <<= 1;
  for (int i = threadIdx.x; i < n; i += blockDim.x)
    keys[i] = i < N ? ((unsigned long long)fkey(scratch[i]) << 32) | (unsigned)i : ~0ull;
  __syncthreads();
  for (int k = 2; k <= n; k <<= 1) {
    for (int j = k >> 1; j > 0; j >>= 1) {
      for (int i = threadIdx.x; i < n; i += blockDim.x) {
        const int ix = i ^ j;
        if (ix > i) {
          const unsigned long long a = keys[i], c = keys[ix];
          if ((a > c) == ((i & k) == 0)) { keys[i] = c; keys[ix] = a; }
        }
      }
      __syncthreads();
    }
  }
  for (int i = threadIdx.x; i < N; i += blockDim.x) {
    perm[i] = (int32_t)(keys[i] & 0xffffffffu);
    if (scores) scores[i] = scratch[i];
  }
}

// Set-up per device, with that device current: the device address of the scratch
// array (in host code the array's name is only a host-side stand-in) and the
// shared-memory opt-in of the ordering kernel.  Only a complete success is kept; a
// failed attempt leaves nothing behind, so the next call on that device tries again.
constexpr int kMaxDevices = 64;
struct DeviceSetup {
  bool ready = false;
  float* scratch = nullptr;
};
DeviceSetup g_setup[kMaxDevices];
std::mutex g_setup_mu;

cudaError_t setup_device(int dev, float** scratch) {
  if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
  std::lock_guard<std::mutex> lock(g_setup_mu);
  DeviceSetup& s = g_setup[dev];
  if (!s.ready) {
    void* p = nullptr;
    cudaError_t err = cudaGetSymbolAddress(&p, g_noalloc_scores);
    if (err == cudaSuccess)
      err = cudaFuncSetAttribute(noalloc_order, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 DKV_NOALLOC_MAX_N * (int)sizeof(unsigned long long));
    if (err != cudaSuccess) {
      (void)cudaGetLastError();   // do not leave the failure to the next unrelated check
      return err;
    }
    s.scratch = static_cast<float*>(p);
    s.ready = true;
  }
  *scratch = s.scratch;
  return cudaSuccess;
}

}  // namespace
}  // namespace dkv

extern "C" dkv_status_t dkv_candidate_order_noalloc(const void* K_bank, const float* base, int32_t m,
                                                    const void* Kc, int32_t N, int32_t d, int32_t dtype,
                                                    const dkv_params_t* params, float* scores_out,
                                                    int32_t* perm_out, void* stream) {
  using namespace dkv;
  if (!Kc || !perm_out || !params || (m > 0 && (!K_bank || !base))) return DKV_ERR_ARG;
  if (dtype != DKV_DTYPE_BF16 && dtype != DKV_DTYPE_FP32) return DKV_ERR_ARG;
  if (N < 1 || N > DKV_NOALLOC_MAX_N || m < 0 || m > 262144 || (d != 64 && d != 128)) return DKV_ERR_SHAPE;
  const dkv_params_t& p = *params;
  if (!(p.tau > 1.0f) || !(p.eps > 0.0f) || !(p.delta > 0.0f) || !(p.sigma >= 0.0f) ||
      !(p.p == 1.0f || p.p == 2.0f || p.p == 4.0f) || !std::isfinite(p.sigma) || !std::isfinite(p.eps))
    return DKV_ERR_ARG;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return DKV_ERR_CUDA;
  float* scratch = nullptr;
  if (setup_device(dev, &scratch) != cudaSuccess) return DKV_ERR_CUDA;
  const float sg = p.sigma > 0.0f ? p.sigma : std::sqrt((float)d / 2.0f);
  KParams kp{};
  kp.inv_s2 = 1.0f / (sg * sg);
  kp.eps = p.eps;
  kp.tau = p.tau;
  kp.delta = p.delta;
  kp.p = (int)p.p;
  kp.sync_heads = 1;
  cudaStream_t s = (cudaStream_t)stream;
  if (m > 0) {
    const dim3 grid((N + ROWS - 1) / ROWS);
    if (dtype == DKV_DTYPE_BF16) {
      using T = __nv_bfloat16;
      if (d == 128) noalloc_score<T, 128><<<grid, ROWS, 0, s>>>((const T*)K_bank, base, m, (const T*)Kc, N, kp, scratch);
      else noalloc_score<T, 64><<<grid, ROWS, 0, s>>>((const T*)K_bank, base, m, (const T*)Kc, N, kp, scratch);
    } else {
      if (d == 128)
        noalloc_score<float, 128><<<grid, ROWS, 0, s>>>((const float*)K_bank, base, m, (const float*)Kc, N, kp, scratch);
      else
        noalloc_score<float, 64><<<grid, ROWS, 0, s>>>((const float*)K_bank, base, m, (const float*)Kc, N, kp, scratch);
    }
    if (cudaGetLastError() != cudaSuccess) return DKV_ERR_CUDA;
  }
  int n = 2;
  while (n < N) n <<= 1;
  noalloc_order<<<1, SORT_THREADS, (size_t)n * sizeof(unsigned long long), s>>>(scratch, N, m, perm_out, scores_out);
  return cudaGetLastError() == cudaSuccess ? DKV_OK : DKV_ERR_CUDA;
}
