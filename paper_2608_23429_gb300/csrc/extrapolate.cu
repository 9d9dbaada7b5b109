// Instantiations of the direct-load kernel (direct_kernel.cuh) without gates.
#include "direct_kernel.cuh"

namespace cbk {
namespace {

template <int K, bool CB16>
cudaError_t launch_k(const ExtrapArgs& a, int grid, cudaStream_t s) {
    extrapolate_kernel<K, CB16, false><<<grid, kThreads, 0, s>>>(a);
    return cudaGetLastError();
}

template <int K, bool CB16>
cudaError_t occ_k(int* blocks) {
    return cudaOccupancyMaxActiveBlocksPerMultiprocessor(blocks, extrapolate_kernel<K, CB16, false>, kThreads, 0);
}

template <bool CB16>
cudaError_t dispatch(const ExtrapArgs& a, int K, int grid, cudaStream_t s) {
    switch (K) {
    case 1: return launch_k<1, CB16>(a, grid, s);
    case 2: return launch_k<2, CB16>(a, grid, s);
    case 3: return launch_k<3, CB16>(a, grid, s);
    case 4: return launch_k<4, CB16>(a, grid, s);
    case 5: return launch_k<5, CB16>(a, grid, s);
    case 6: return launch_k<6, CB16>(a, grid, s);
    case 7: return launch_k<7, CB16>(a, grid, s);
    case 8: return launch_k<8, CB16>(a, grid, s);
    default: return cudaErrorInvalidValue;
    }
}

template <bool CB16>
cudaError_t occupancy(int K, int* blocks) {
    switch (K) {
    case 1: return occ_k<1, CB16>(blocks);
    case 2: return occ_k<2, CB16>(blocks);
    case 3: return occ_k<3, CB16>(blocks);
    case 4: return occ_k<4, CB16>(blocks);
    case 5: return occ_k<5, CB16>(blocks);
    case 6: return occ_k<6, CB16>(blocks);
    case 7: return occ_k<7, CB16>(blocks);
    case 8: return occ_k<8, CB16>(blocks);
    default: return cudaErrorInvalidValue;
    }
}

}  // namespace

cudaError_t launch_extrapolate(const ExtrapArgs& a, int K, bool cache_bf16, int grid, cudaStream_t s) {
    return cache_bf16 ? dispatch<true>(a, K, grid, s) : dispatch<false>(a, K, grid, s);
}

cudaError_t extrapolate_blocks_per_sm(int K, bool cache_bf16, int* blocks) {
    return cache_bf16 ? occupancy<true>(K, blocks) : occupancy<false>(K, blocks);
}

}  // namespace cbk
