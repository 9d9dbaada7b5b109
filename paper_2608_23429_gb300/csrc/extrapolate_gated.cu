// Instantiations of the direct-load kernel (direct_kernel.cuh) with
// per-(batch, channel) gates on the hidden-state update.
#include "direct_kernel.cuh"

namespace cbk {
namespace {

template <int K, bool CB16>
cudaError_t launch_gk(const ExtrapArgs& a, int grid, cudaStream_t s) {
    extrapolate_kernel<K, CB16, true><<<grid, kThreads, 0, s>>>(a);
    return cudaGetLastError();
}

template <bool CB16>
cudaError_t dispatch_g(const ExtrapArgs& a, int K, int grid, cudaStream_t s) {
    switch (K) {
    case 1: return launch_gk<1, CB16>(a, grid, s);
    case 2: return launch_gk<2, CB16>(a, grid, s);
    case 3: return launch_gk<3, CB16>(a, grid, s);
    case 4: return launch_gk<4, CB16>(a, grid, s);
    case 5: return launch_gk<5, CB16>(a, grid, s);
    case 6: return launch_gk<6, CB16>(a, grid, s);
    case 7: return launch_gk<7, CB16>(a, grid, s);
    case 8: return launch_gk<8, CB16>(a, grid, s);
    default: return cudaErrorInvalidValue;
    }
}

}  // namespace

cudaError_t launch_extrapolate_gated(const ExtrapArgs& a, int K, bool cache_bf16, int grid, cudaStream_t s) {
    return cache_bf16 ? dispatch_g<true>(a, K, grid, s) : dispatch_g<false>(a, K, grid, s);
}

}  // namespace cbk
