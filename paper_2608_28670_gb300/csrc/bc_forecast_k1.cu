// bc_forecast_k1.cu -- the grouped forecast kernels and their launcher for windows of
// H = 1 nodes (Eq. 13 with 1 terms); the kernels themselves are in bc_forecast_kernels.cuh.
#include "bc_forecast_kernels.cuh"

namespace bc {

int launch_forecast_k1(const LaunchPlan &plan, void *stream, int64_t *launches,
                       int64_t *pipeline_launches) {
    return dispatch_dtypes<1>(plan, static_cast<cudaStream_t>(stream), launches,
                              pipeline_launches);
}

}  // namespace bc
