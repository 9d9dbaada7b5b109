// Skipped-step kernel, direct-load variant: f_t = sum_j w_j f_{s_j} for every
// cached branch tensor (Sec. 3.3, Eq. for f_t; Alg. 1, extrapolation branch),
// optionally added into the block's hidden state (Sec. 3.1, B(x) = x + S + C + M).
//
// A K-term streaming reduction (K reads and one write per element against
// ~2K flops) is HBM-bound, so the kernel is shaped for bandwidth:
//   * one persistent grid covers every tensor of every block; tiles of 4096
//     (bf16) or 2048 (fp32) elements are dealt round-robin to the CTAs, and
//     each CTA walks its item table forward, so no search is needed;
//   * every thread issues all of its K x 16-B plain global loads (bf16: two
//     8-element vectors, fp32: one) before any arithmetic;
//   * the weights arrive as kernel parameters (fp32 high/low pairs).
// The arithmetic is in cb_math.cuh. The bulk-copy pipeline variant
// (bulk_kernel.cuh) computes the same bits from shared memory. GATED: the
// hidden states receive g_b * P_b (per-(batch, channel) gates); instantiated
// in extrapolate_gated.cu, the un-gated kernels in extrapolate.cu.
#pragma once

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
            const unsigned char* p = hist_ptr(A, j, moff) + ev[u] * ES;
            raw[u][j][0] = ld_v4(p);
            if constexpr (!CB16) raw[u][j][CB16 ? 0 : 1] = ld_v4(p + 16);
        }
}

template <int K, bool CB16, int UV, bool GATED>
__device__ __forceinline__ void item_vectors(const ExtrapArgs& A, int it, const long long (&ev)[UV]) {
    const int nb = A.nb[it];
    const int first = A.first[it];
    void* resid = A.resid[it];
    unsigned gi[UV];
    if constexpr (GATED) {  // items without shapes carry no gate
        if (A.i_hidden[it] != 0) gate_offsets<UV>(A, it, ev[0], ev, gi);
    }
    if (A.precise) {
        Acc<UV> acc;
        acc.zero();
        for (int m = 0; m < nb; ++m) {
            RawVecs<K, CB16, UV> raw;
            load_member<K, CB16, UV>(A, A.m_off[first + m], ev, raw);
            void* out = member_out<K, CB16, UV>(A, first + m, ev, raw);
            if constexpr (GATED) {
                float g[UV][8];
                load_gates<UV>(A, first + m, gi, g);
                member_precise<K, CB16, UV, true>(A, out, ev, raw, resid != nullptr, acc,
                                                  [&](int u, float (&gv)[8]) {
#pragma unroll
                                                      for (int e = 0; e < 8; ++e) gv[e] = g[u][e];
                                                  });
            } else {
                member_precise<K, CB16, UV>(A, out, ev, raw, resid != nullptr, acc);
            }
        }
        if (resid)
            resid_precise<UV>(A, ev, acc, resid, [&](int u, float (&x)[8]) { load_x8(resid, A.resid_bf16, ev[u], x); });
    } else {
        Acc<UV> acc;
        acc.zero();
        for (int m = 0; m < nb; ++m) {
            RawVecs<K, CB16, UV> raw;
            load_member<K, CB16, UV>(A, A.m_off[first + m], ev, raw);
            void* out = member_out<K, CB16, UV>(A, first + m, ev, raw);
            // full-step epilogue from bf16 features: exact features, no weighted
            // sum (the bulk kernel's ONE path; from fp32 features both kernels
            // take the general path)
            bool one = false;
            if constexpr (K == 1 && CB16) {
                one = A.copy_out != 0;
                if (one && resid) {
                    if constexpr (GATED) {
                        float g[UV][8];
                        load_gates<UV>(A, first + m, gi, g);
                        member_one<K, CB16, UV, true>(raw, acc, [&](int u, float (&gv)[8]) {
#pragma unroll
                            for (int e = 0; e < 8; ++e) gv[e] = g[u][e];
                        });
                    } else {
                        member_one<K, CB16, UV>(raw, acc);
                    }
                }
            }
            if (one) {
            } else if constexpr (GATED) {
                float g[UV][8];
                load_gates<UV>(A, first + m, gi, g);
                member_fast<K, CB16, UV, false, true>(A, A.m_off[first + m], out, ev, raw,
                                                      resid != nullptr, acc, [&](int u, float (&gv)[8]) {
#pragma unroll
                                                          for (int e = 0; e < 8; ++e) gv[e] = g[u][e];
                                                      });
            } else {
                member_fast<K, CB16, UV, false>(A, A.m_off[first + m], out, ev, raw,
                                                resid != nullptr, acc);
            }
        }
        if (resid)
            resid_fast<K, UV>(
                A, it, ev, acc, resid, [&](int u, float (&x)[8]) { load_x8(resid, true, ev[u], x); },
                [&](int u, int e, float xe, float& hi, float& lo) {
                    exact_resid<CB16>(A, K, it, ev[u] + e, xe, hi, lo);
                },
                // member_one's sums are unscaled (bf16 epilogue); member_fast's are scaled
                (K == 1 && CB16 && A.copy_out) ? A.w_guard[0] : 1.0f);
    }
}

template <int K, bool CB16, bool GATED>
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
            item_vectors<K, CB16, U, GATED>(A, it, ev);
        } else if (A.vec_ok[it]) {  // the ragged last tile of an aligned item
            for (int u = 0; u < U; ++u) {
                const long long v0 = e0 + ((long long)u * kThreads + threadIdx.x) * kVecElems;
                if (v0 + kVecElems <= numel) {
                    const long long ev1[1] = {v0};
                    item_vectors<K, CB16, 1, GATED>(A, it, ev1);
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

}  // namespace
}  // namespace cbk
