// Instantiations of the bulk-copy pipeline kernel (bulk_kernel.cuh) without
// gates: prediction-only launches and launches that add the predictions
// straight into the hidden states.
#include "bulk_kernel.cuh"

namespace cbk {
namespace {

template <int K, bool CB16>
cudaError_t launch_k(const ExtrapArgs& a, bool grouped, int grid, size_t smem, cudaStream_t s) {
    if (grouped)
        extrapolate_bulk_kernel<K, CB16, true, false><<<grid, Shape<CB16, K, true, false>::threads, smem, s>>>(a);
    else
        extrapolate_bulk_kernel<K, CB16, false, false><<<grid, Shape<CB16, K, false, false>::threads, smem, s>>>(a);
    return cudaGetLastError();
}

template <int K, bool CB16>
cudaError_t prepare_k(size_t smem) {
    cudaError_t e = cudaFuncSetAttribute(extrapolate_bulk_kernel<K, CB16, true, false>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    return cudaFuncSetAttribute(extrapolate_bulk_kernel<K, CB16, false, false>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                (int)smem);
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
