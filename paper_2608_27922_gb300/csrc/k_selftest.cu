// Self-test of the bounded device-side waits: one CTA waits, through the same helper as
// every tensor-core kernel, on an mbarrier that nothing ever arrives on, gives up after
// the requested limit, records the timeout in its error word and returns, so the
// context stays usable.  No fault, trap or hang is involved.
#include "dkv.h"
#include "dkv_internal.h"
#include "tc_ptx.cuh"

namespace dkv {
namespace {

using namespace tc;

__global__ void k_wait_timeout(uint64_t limit_ns, int32_t* err, int64_t* elapsed_ns) {
  __shared__ __align__(8) uint64_t bar;
  __shared__ int abort_flag;
  if (threadIdx.x == 0) {
    mbar_init(&bar, 1);   // one arrival expected; nothing ever arrives
    abort_flag = 0;
    fence_barrier_init();
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    const uint64_t t0 = globaltimer_ns();
    const bool ok = mbar_wait_limit(&bar, 0, reinterpret_cast<volatile int*>(&abort_flag), limit_ns);
    *elapsed_ns = (int64_t)(globaltimer_ns() - t0);
    *err = ok ? DEV_OK : DEV_TIMEOUT;
  }
}

}  // namespace
}  // namespace dkv

extern "C" dkv_status_t dkv_selftest_wait_timeout(int32_t limit_us, int64_t* elapsed_ns) {
  using namespace dkv;
  if (limit_us < 1 || limit_us > 1000000 || !elapsed_ns) return DKV_ERR_ARG;
  int32_t* d_err = nullptr;
  int64_t* d_el = nullptr;
  if (cudaMalloc(&d_err, sizeof(int32_t)) != cudaSuccess) return DKV_ERR_NOMEM;
  if (cudaMalloc(&d_el, sizeof(int64_t)) != cudaSuccess) {
    cudaFree(d_err);
    return DKV_ERR_NOMEM;
  }
  int32_t err = -1;
  int64_t el = 0;
  k_wait_timeout<<<1, 32>>>((uint64_t)limit_us * 1000ull, d_err, d_el);
  cudaError_t e = cudaGetLastError();
  if (e == cudaSuccess) e = cudaDeviceSynchronize();
  if (e == cudaSuccess) e = cudaMemcpy(&err, d_err, sizeof(err), cudaMemcpyDeviceToHost);
  if (e == cudaSuccess) e = cudaMemcpy(&el, d_el, sizeof(el), cudaMemcpyDeviceToHost);
  cudaFree(d_err);
  cudaFree(d_el);
  if (e != cudaSuccess) return DKV_ERR_CUDA;
  *elapsed_ns = el;
  return err == DEV_TIMEOUT ? DKV_ERR_TIMEOUT : (err == DEV_OK ? DKV_OK : DKV_ERR_DEVICE);
}
