// Skipped-step kernel, direct-load variant: f_t = sum_j w_j f_{s_j} for every
// cached branch tensor (Sec. 3.3, Eq. for f_t; Alg. 1, extrapolation branch),
// optionally added into the block's hidden state (Sec. 3.1, B(x) = x + S + C + M).
//
// A K-term streaming reduction (K reads and one write per element against
// ~2K flops) is HBM-bound, so the kernel is shaped for bandwidth:
//   * one persistent grid covers every tensor of every block; tiles of 4096
//     (bf16) or 2048 (fp32) elements are dealt round-robin to the CTAs, and
//     each CTA walks its item table forward, so no search is needed;
//   * every thread issues all of its K x 16-B non-coherent, L1-bypassing loads
//     (bf16: two 8-element vectors, fp32: one) before any arithmetic;
//   * the weights arrive as kernel parameters (fp32 high/low pairs).
// The arithmetic is in cb_math.cuh. The bulk-copy pipeline variant
// (extrapolate_bulk.cu) computes the same bits from shared memory.
#include "cb_math.cuh"

namespace cbk {
namespace {

template <int K, bool CB16, int UV>
__device__ __forceinline__ void load_member(const ExtrapArgs& A, long long moff, const long long (&ev)[UV],
                                            RawVecs<K, CB16, UV>& raw) {
    constexpr int ES = CB16 ? 2 : 4;
#pragma unroll
    for (int u = 0; u < UV; ++u)
#pragma unroll
        for (int j = 0; j < K; ++j) {
            const unsigned char* p = A.cache + A.slot_off[j] + moff + ev[u] * ES;
            raw[u][j][0] = ld_stream(p);
            if constexpr (!CB16) raw[u][j][CB16 ? 0 : 1] = ld_stream(p + 16);
        }
}

template <int K, bool CB16, int UV>
__device__ __forceinline__ void item_vectors(const ExtrapArgs& A, int it, const long long (&ev)[UV]) {
    const int nb = A.nb[it];
    const int first = A.first[it];
    void* resid = A.resid[it];
    if (A.precise) {
        Acc<UV> acc;
        acc.zero();
        for (int m = 0; m < nb; ++m) {
            RawVecs<K, CB16, UV> raw;
            load_member<K, CB16, UV>(A, A.m_off[first + m], ev, raw);
            member_precise<K, CB16, UV>(A, A.m_out[first + m], ev, raw, resid != nullptr, acc);
        }
        if (resid)
            resid_precise<UV>(A, ev, acc, resid, [&](int u, float (&x)[8]) { load_x8(resid, A.resid_bf16, ev[u], x); });
    } else {
        Acc<UV> acc;
        acc.zero();
        for (int m = 0; m < nb; ++m) {
            RawVecs<K, CB16, UV> raw;
            load_member<K, CB16, UV>(A, A.m_off[first + m], ev, raw);
            member_fast<K, CB16, UV, false>(A, A.m_off[first + m], A.m_out[first + m], ev, raw, resid != nullptr,
                                            acc);
        }
        if (resid)
            resid_fast<K, UV>(
                A, it, ev, acc, resid, [&](int u, float (&x)[8]) { load_x8(resid, true, ev[u], x); },
                [&](int u, int e, float xe, float& hi, float& lo) {
                    exact_resid<CB16>(A, K, it, ev[u] + e, xe, hi, lo);
                });
    }
}

template <int K, bool CB16>
__global__ void __launch_bounds__(kThreads) extrapolate_kernel(const __grid_constant__ ExtrapArgs A) {
    constexpr int U = vectors_per_thread(CB16);
    constexpr long long TE = tile_elems(CB16);
    int it = 0;
    for (int tile = blockIdx.x; tile < A.tiles_total; tile += gridDim.x) {
        while (tile >= A.tile_begin[it + 1]) ++it;  // tiles only grow: walk forward
        const long long numel = A.numel[it];
        const long long e0 = (long long)(tile - A.tile_begin[it]) * TE;
        if (A.vec_ok[it] && e0 + TE <= numel) {
            long long ev[U];
#pragma unroll
            for (int u = 0; u < U; ++u) ev[u] = e0 + ((long long)u * kThreads + threadIdx.x) * kVecElems;
            item_vectors<K, CB16, U>(A, it, ev);
        } else if (A.vec_ok[it]) {  // the ragged last tile of an aligned item
            for (int u = 0; u < U; ++u) {
                const long long v0 = e0 + ((long long)u * kThreads + threadIdx.x) * kVecElems;
                if (v0 + kVecElems <= numel) {
                    const long long ev1[1] = {v0};
                    item_vectors<K, CB16, 1>(A, it, ev1);
                } else {
                    for (long long e = v0; e < numel; ++e) scalar_element<CB16>(A, K, it, e);
                }
            }
        } else {  // misaligned item: element-wise, adjacent threads on adjacent elements
            const long long end = e0 + TE < numel ? e0 + TE : numel;
            for (long long e = e0 + threadIdx.x; e < end; e += kThreads) scalar_element<CB16>(A, K, it, e);
        }
    }
}

template <int K, bool CB16>
cudaError_t launch_k(const ExtrapArgs& a, int grid, cudaStream_t s) {
    extrapolate_kernel<K, CB16><<<grid, kThreads, 0, s>>>(a);
    return cudaGetLastError();
}

template <int K, bool CB16>
cudaError_t occ_k(int* blocks) {
    return cudaOccupancyMaxActiveBlocksPerMultiprocessor(blocks, extrapolate_kernel<K, CB16>, kThreads, 0);
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
