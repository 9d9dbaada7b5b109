// Instantiations of the bulk-copy pipeline kernel (bulk_kernel.cuh) with
// per-(batch, channel) gates on the hidden-state update: x <- x + sum_b g_b P_b.
#include "bulk_kernel.cuh"

namespace cbk {
namespace {

// The full-step epilogue from bf16 features (a copy_out launch without
// compensated hidden states) runs the ONE instantiation; from fp32 features
// the general path (see extrapolate_bulk.cu).
template <int K, bool CB16>
cudaError_t launch_gk(const ExtrapArgs& a, int grid, size_t smem, cudaStream_t s) {
    if constexpr (K == 1 && CB16) {
        if (a.copy_out && !a.precise) {
            extrapolate_bulk_kernel<K, CB16, true, true, true><<<grid, Shape<CB16, K, true, true>::threads, smem, s>>>(a);
            return cudaGetLastError();
        }
    }
    extrapolate_bulk_kernel<K, CB16, true, true><<<grid, Shape<CB16, K, true, true>::threads, smem, s>>>(a);
    return cudaGetLastError();
}

template <int K, bool CB16>
cudaError_t prepare_gk(size_t smem) {
    cudaError_t e = cudaFuncSetAttribute(extrapolate_bulk_kernel<K, CB16, true, true>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if constexpr (K == 1 && CB16)
        if (e == cudaSuccess)
            e = cudaFuncSetAttribute(extrapolate_bulk_kernel<K, CB16, true, true, true>,
                                     cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    return e;
}

#define CB_K_SWITCH(K, CALL)                  \
    switch (K) {                              \
    case 1: return CALL(1);                   \
    case 2: return CALL(2);                   \
    case 3: return CALL(3);                   \
    case 4: return CALL(4);                   \
    case 5: return CALL(5);                   \
    case 6: return CALL(6);                   \
    case 7: return CALL(7);                   \
    case 8: return CALL(8);                   \
    default: return cudaErrorInvalidValue;    \
    }

}  // namespace

cudaError_t prepare_extrapolate_bulk_gated(int K, bool cache_bf16, size_t smem) {
#define P_BF(k) prepare_gk<k, true>(smem)
#define P_F32(k) prepare_gk<k, false>(smem)
    if (cache_bf16) {
        CB_K_SWITCH(K, P_BF)
    }
    CB_K_SWITCH(K, P_F32)
#undef P_BF
#undef P_F32
}

cudaError_t launch_extrapolate_bulk_gated(const ExtrapArgs& a, int K, bool cache_bf16, int grid, size_t smem,
                                          cudaStream_t s) {
#define L_BF(k) launch_gk<k, true>(a, grid, smem, s)
#define L_F32(k) launch_gk<k, false>(a, grid, smem, s)
    if (cache_bf16) {
        CB_K_SWITCH(K, L_BF)
    }
    CB_K_SWITCH(K, L_F32)
#undef L_BF
#undef L_F32
}

}  // namespace cbk
