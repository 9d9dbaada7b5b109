// Instantiations of the bulk-copy pipeline kernel (bulk_kernel.cuh) without
// gates: prediction-only launches and launches that add the predictions
// straight into the hidden states.
#include "bulk_kernel.cuh"

namespace cbk {
namespace {

template <int K, bool CB16, bool ONE>
cudaError_t launch_kk(const ExtrapArgs& a, bool grouped, int grid, size_t smem, cudaStream_t s) {
    if (grouped)
        extrapolate_bulk_kernel<K, CB16, true, false, ONE><<<grid, Shape<CB16, K, true, false>::threads, smem, s>>>(a);
    else
        extrapolate_bulk_kernel<K, CB16, false, false, ONE><<<grid, Shape<CB16, K, false, false>::threads, smem, s>>>(a);
    return cudaGetLastError();
}

// The full-step epilogue from bf16 features (a copy_out launch without
// compensated hidden states) runs the ONE instantiations. From fp32 features
// the general path measured faster on GB300 (FLUX 95.6 % against 89.0 % of the
// copy peak), so those launches keep it.
template <int K, bool CB16>
cudaError_t launch_k(const ExtrapArgs& a, bool grouped, int grid, size_t smem, cudaStream_t s) {
    if constexpr (K == 1 && CB16)
        if (a.copy_out && !a.precise) return launch_kk<K, CB16, true>(a, grouped, grid, smem, s);
    return launch_kk<K, CB16, false>(a, grouped, grid, smem, s);
}

template <int K, bool CB16, bool ONE>
cudaError_t prepare_kk(size_t smem) {
    cudaError_t e = cudaFuncSetAttribute(extrapolate_bulk_kernel<K, CB16, true, false, ONE>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    return cudaFuncSetAttribute(extrapolate_bulk_kernel<K, CB16, false, false, ONE>,
                                cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
}

template <int K, bool CB16>
cudaError_t prepare_k(size_t smem) {
    cudaError_t e = prepare_kk<K, CB16, false>(smem);
    if constexpr (K == 1 && CB16)
        if (e == cudaSuccess) e = prepare_kk<K, CB16, true>(smem);
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

size_t bulk_smem_bytes(int chunks_per_stage, size_t extra_per_stage, int stages) {
    return kBarrierBytes + (size_t)stages * ((size_t)chunks_per_stage * kChunkBytes + extra_per_stage);
}

cudaError_t prepare_extrapolate_bulk(int K, bool cache_bf16, size_t smem) {
#define P_BF(k) prepare_k<k, true>(smem)
#define P_F32(k) prepare_k<k, false>(smem)
    if (cache_bf16) {
        CB_K_SWITCH(K, P_BF)
    }
    CB_K_SWITCH(K, P_F32)
#undef P_BF
#undef P_F32
}

cudaError_t launch_extrapolate_bulk(const ExtrapArgs& a, int K, bool cache_bf16, bool grouped, int grid, size_t smem,
                                    cudaStream_t s) {
#define L_BF(k) launch_k<k, true>(a, grouped, grid, smem, s)
#define L_F32(k) launch_k<k, false>(a, grouped, grid, smem, s)
    if (cache_bf16) {
        CB_K_SWITCH(K, L_BF)
    }
    CB_K_SWITCH(K, L_F32)
#undef L_BF
#undef L_F32
}

}  // namespace cbk
