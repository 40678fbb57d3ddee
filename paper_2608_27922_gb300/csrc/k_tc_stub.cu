// Placeholder for the tcgen05 kernels: reports "not supported" so the
// tensor-core score mode is refused at create time.
#include "dkv_internal.h"

namespace dkv {
bool tc_supported(int, int) { return false; }
cudaError_t tc_set_smem_limits() { return cudaSuccess; }
cudaError_t launch_score_tc(const Bank&, const Ws&, const void*, int, const KParams&, cudaStream_t, Timer*) { return cudaErrorNotSupported; }
cudaError_t launch_cross_tc(const Bank&, const Ws&, const KParams&, cudaStream_t, Timer*) { return cudaErrorNotSupported; }
cudaError_t launch_project_tc(const Bank&, const Ws&, const KParams&, cudaStream_t, Timer*) { return cudaErrorNotSupported; }
cudaError_t launch_subtract_tc(const Bank&, const Ws&, const KParams&, cudaStream_t, Timer*) { return cudaErrorNotSupported; }
cudaError_t launch_newbase_tc(const Bank&, const Ws&, const KParams&, cudaStream_t, Timer*) { return cudaErrorNotSupported; }
cudaError_t launch_attend_tc(const Bank&, const void*, int, const void*, const void*, int, void*, cudaStream_t, Timer*) { return cudaErrorNotSupported; }
}  // namespace dkv
