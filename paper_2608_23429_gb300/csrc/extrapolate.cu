// Skipped-step kernel: f_t = sum_j w_j f_{s_j} for every cached branch tensor
// (Sec. 3.3, Eq. for f_t; Alg. 1, extrapolation branch), optionally added into
// the block's hidden state (Sec. 3.1, B(x) = x + S + C + M).
//
// The work is a K-term streaming reduction: K reads and one write per element
// against ~2K flops, i.e. far below any compute ridge, so the kernel is shaped
// for HBM bandwidth, not tensor cores:
//   * one persistent grid covers every tensor of every block; tiles of 4096
//     (bf16) or 2048 (fp32) elements are dealt round-robin to the CTAs, and
//     each CTA walks its item table forward, so no search is needed;
//   * every thread issues all of its K x 16-B (bf16: 2 vectors, fp32: 1
//     vector of 32 B) non-coherent, L1-bypassing loads before any arithmetic,
//     keeping 2K independent 16-B requests in flight per thread;
//   * the weights arrive as kernel parameters (fp32 high/low pairs), so there
//     is no host-to-device copy on the hot path.
//
// Arithmetic. The fast path accumulates s = sum_j w_hi[j] F_j with fp32 FMAs
// and, alongside, a = sum_j |w_hi[j]| |F_j|. With unit roundoff u = 2^-24 the
// FMA chain and the dropped low weight half give |s - P| <= (K+1) u a (1+O(Ku)),
// so whenever (K+2) u a <= 2^-10 |s| the error is below a quarter of a bf16
// spacing and bf16(s) is within one bf16 ulp of bf16(P). Elements that fail
// this test (strong cancellation, rare) and every element of an fp32 result
// are computed with Ogita, Rump & Oishi's Dot2 (SIAM J. Sci. Comput. 26(6),
// 2005: TwoProduct by FMA plus TwoSum), which carries the result as an
// unevaluated pair hi + lo and is then rounded once to the output type.
#include <cuda_bf16.h>

#include "cb_device.h"

namespace cbk {
namespace {

constexpr float kU = 0x1.0p-24f;

__device__ __forceinline__ uint4 ld_stream(const unsigned char* p) {
    uint4 v;
    asm("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
        : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
        : "l"(p));
    return v;
}

__device__ __forceinline__ void unpack_bf16x8(const uint4& v, float (&f)[8]) {
    const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        f[2 * i] = __uint_as_float(w[i] << 16);
        f[2 * i + 1] = __uint_as_float(w[i] & 0xFFFF0000u);
    }
}

__device__ __forceinline__ void unpack_f32x8(const uint4& a, const uint4& b, float (&f)[8]) {
    f[0] = __uint_as_float(a.x); f[1] = __uint_as_float(a.y);
    f[2] = __uint_as_float(a.z); f[3] = __uint_as_float(a.w);
    f[4] = __uint_as_float(b.x); f[5] = __uint_as_float(b.y);
    f[6] = __uint_as_float(b.z); f[7] = __uint_as_float(b.w);
}

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
    __nv_bfloat162 h = __floats2bfloat162_rn(lo, hi);  // RNE; .x is the low half
    return *reinterpret_cast<uint32_t*>(&h);
}

__device__ __forceinline__ uint16_t bf16_bits(float x) {
    return __bfloat16_as_ushort(__float2bfloat16_rn(x));
}

// ---- error-free transformations (all operations explicitly rounded, never contracted)
__device__ __forceinline__ void two_sum(float a, float b, float& s, float& e) {
    s = __fadd_rn(a, b);
    const float bb = __fsub_rn(s, a);
    e = __fadd_rn(__fsub_rn(a, __fsub_rn(s, bb)), __fsub_rn(b, bb));
}

// One Dot2 term: (p, c) += (w_hi + w_lo) * f, p the running sum, c its error.
__device__ __forceinline__ void dot2_step(float w_hi, float w_lo, float f, float& p, float& c) {
    const float h = __fmul_rn(w_hi, f);
    const float r = __fmaf_rn(w_hi, f, -h);  // exact: w_hi*f - h
    float q;
    two_sum(p, h, p, q);
    c = __fadd_rn(c, __fadd_rn(q, r));
    c = __fmaf_rn(w_lo, f, c);
}

// bf16 of the exact value hi + lo, where hi = fl(hi + lo) (so |lo| <= ulp(hi)/2).
// Only when hi sits exactly on a bf16 rounding midpoint can lo change the
// outcome; then the sign of lo decides, otherwise hi rounds like hi + lo.
__device__ __forceinline__ uint16_t bf16_of_pair(float hi, float lo) {
    const uint32_t b = __float_as_uint(hi);
    if ((b & 0xFFFFu) == 0x8000u && lo != 0.0f && (b & 0x7F800000u) != 0x7F800000u) {
        const bool away = (lo > 0.0f) == (hi > 0.0f);
        return (uint16_t)((b >> 16) + (away ? 1u : 0u));
    }
    return bf16_bits(hi);
}

template <bool CB16>
__device__ __forceinline__ float load_cache_elem(const unsigned char* base, long long e) {
    if constexpr (CB16) {
        const uint16_t h = reinterpret_cast<const uint16_t*>(base)[e];
        return __uint_as_float((uint32_t)h << 16);
    } else {
        return reinterpret_cast<const float*>(base)[e];
    }
}

__device__ __forceinline__ float load_elem(const void* p, bool bf16, long long e) {
    if (bf16) return __uint_as_float((uint32_t)(reinterpret_cast<const uint16_t*>(p)[e]) << 16);
    return reinterpret_cast<const float*>(p)[e];
}

__device__ __forceinline__ void store_pair(void* p, bool bf16, long long e, float hi, float lo) {
    if (bf16)
        reinterpret_cast<uint16_t*>(p)[e] = bf16_of_pair(hi, lo);
    else
        reinterpret_cast<float*>(p)[e] = hi;
}

// Compensated value of member tensor (byte offset moff) at element e.
template <bool CB16>
__device__ __noinline__ void exact_member(const ExtrapArgs& A, int K, long long moff, long long e,
                                          float& hi, float& lo) {
    float p = 0.0f, c = 0.0f;
    for (int j = 0; j < K; ++j) {
        const float f = load_cache_elem<CB16>(A.cache + A.slot_off[j] + moff, e);
        dot2_step(A.w_hi[j], A.w_lo[j], f, p, c);
    }
    two_sum(p, c, hi, lo);
}

// Compensated hidden-state update of item `it` at element e: x + sum_b P_b.
template <bool CB16>
__device__ __noinline__ void exact_resid(const ExtrapArgs& A, int K, int it, long long e, float x,
                                         float& hi, float& lo) {
    float tp = x, tc = 0.0f;
    const int first = A.first[it];
    for (int m = 0; m < A.nb[it]; ++m) {
        float h, l, q;
        exact_member<CB16>(A, K, A.m_off[first + m], e, h, l);
        two_sum(tp, h, tp, q);
        tc = __fadd_rn(tc, __fadd_rn(q, l));
    }
    two_sum(tp, tc, hi, lo);
}

// One element through the compensated path (misaligned items and ragged tails).
template <bool CB16>
__device__ __noinline__ void scalar_element(const ExtrapArgs& A, int K, int it, long long e) {
    const int first = A.first[it];
    void* resid = A.resid[it];
    float tp = 0.0f, tc = 0.0f;
    for (int m = 0; m < A.nb[it]; ++m) {
        float hi, lo, q;
        exact_member<CB16>(A, K, A.m_off[first + m], e, hi, lo);
        if (A.m_out[first + m]) store_pair(A.m_out[first + m], A.out_bf16, e, hi, lo);
        two_sum(tp, hi, tp, q);
        tc = __fadd_rn(tc, __fadd_rn(q, lo));
    }
    if (resid) {
        float q, hi, lo;
        two_sum(tp, load_elem(resid, A.resid_bf16, e), tp, q);
        tc = __fadd_rn(tc, q);
        two_sum(tp, tc, hi, lo);
        store_pair(resid, A.resid_bf16, e, hi, lo);
    }
}

template <int K, bool CB16, int UV>
__device__ __forceinline__ void load_member(const ExtrapArgs& A, long long moff, const long long (&ev)[UV],
                                            uint4 (&raw)[UV][K][CB16 ? 1 : 2]) {
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

template <bool CB16>
__device__ __forceinline__ void unpack(const uint4 (&r)[CB16 ? 1 : 2], float (&f)[8]) {
    if constexpr (CB16)
        unpack_bf16x8(r[0], f);
    else
        unpack_f32x8(r[0], r[CB16 ? 0 : 1], f);
}

__device__ __forceinline__ void load_x8(const void* p, bool bf16, long long e, float (&x)[8]) {
    if (bf16) {
        const uint4 v = *reinterpret_cast<const uint4*>(reinterpret_cast<const uint16_t*>(p) + e);
        unpack_bf16x8(v, x);
    } else {
        const uint4* q = reinterpret_cast<const uint4*>(reinterpret_cast<const float*>(p) + e);
        unpack_f32x8(q[0], q[1], x);
    }
}

__device__ __forceinline__ void store_bf16x8(void* p, long long e, const uint32_t (&pk)[4]) {
    *reinterpret_cast<uint4*>(reinterpret_cast<uint16_t*>(p) + e) = make_uint4(pk[0], pk[1], pk[2], pk[3]);
}

__device__ __forceinline__ void store_f32x8(void* p, long long e, const float (&v)[8]) {
    uint4* q = reinterpret_cast<uint4*>(reinterpret_cast<float*>(p) + e);
    q[0] = make_uint4(__float_as_uint(v[0]), __float_as_uint(v[1]), __float_as_uint(v[2]), __float_as_uint(v[3]));
    q[1] = make_uint4(__float_as_uint(v[4]), __float_as_uint(v[5]), __float_as_uint(v[6]), __float_as_uint(v[7]));
}

__device__ __forceinline__ void set_half(uint32_t (&pk)[4], int e, uint16_t h) {
    uint32_t& w = pk[e >> 1];
    w = (e & 1) ? ((w & 0x0000FFFFu) | ((uint32_t)h << 16)) : ((w & 0xFFFF0000u) | h);
}

// Fast path over UV aligned 8-element vectors: fp32 FMA with a guarded
// compensated fallback. Only reached with bf16 predictions and hidden states.
template <int K, bool CB16, int UV>
__device__ __forceinline__ void vec_fast(const ExtrapArgs& A, int it, const long long (&ev)[UV]) {
    const int nb = A.nb[it];
    const int first = A.first[it];
    void* resid = A.resid[it];
    const float g_out = (float)(K + 2) * kU * 1.01f;
    float tot[UV][8], tota[UV][8];
#pragma unroll
    for (int u = 0; u < UV; ++u)
#pragma unroll
        for (int e = 0; e < 8; ++e) tot[u][e] = tota[u][e] = 0.0f;

    for (int m = 0; m < nb; ++m) {
        const long long moff = A.m_off[first + m];
        void* out = A.m_out[first + m];
        uint4 raw[UV][K][CB16 ? 1 : 2];
        load_member<K, CB16, UV>(A, moff, ev, raw);
#pragma unroll
        for (int u = 0; u < UV; ++u) {
            float s[8], a[8];
#pragma unroll
            for (int e = 0; e < 8; ++e) s[e] = a[e] = 0.0f;
#pragma unroll
            for (int j = 0; j < K; ++j) {
                float f[8];
                unpack<CB16>(raw[u][j], f);
#pragma unroll
                for (int e = 0; e < 8; ++e) {
                    s[e] = fmaf(A.w_hi[j], f[e], s[e]);
                    a[e] = fmaf(A.w_abs[j], fabsf(f[e]), a[e]);
                }
            }
            if (out) {
                uint32_t pk[4];
#pragma unroll
                for (int i = 0; i < 4; ++i) pk[i] = pack_bf16x2(s[2 * i], s[2 * i + 1]);
#pragma unroll
                for (int e = 0; e < 8; ++e) {
                    if (!(g_out * a[e] <= 0x1.0p-10f * fabsf(s[e]))) {
                        float hi, lo;
                        exact_member<CB16>(A, K, moff, ev[u] + e, hi, lo);
                        set_half(pk, e, bf16_of_pair(hi, lo));
                    }
                }
                store_bf16x8(out, ev[u], pk);
            }
            if (resid) {
#pragma unroll
                for (int e = 0; e < 8; ++e) {
                    tot[u][e] += s[e];
                    tota[u][e] += a[e];
                }
            }
        }
    }
    if (resid) {
        const float g_res = (float)(K + nb + 3) * kU * 1.01f;
#pragma unroll
        for (int u = 0; u < UV; ++u) {
            float x[8];
            load_x8(resid, true, ev[u], x);
            float t[8];
            uint32_t pk[4];
#pragma unroll
            for (int e = 0; e < 8; ++e) t[e] = tot[u][e] + x[e];
#pragma unroll
            for (int i = 0; i < 4; ++i) pk[i] = pack_bf16x2(t[2 * i], t[2 * i + 1]);
#pragma unroll
            for (int e = 0; e < 8; ++e) {
                if (!(g_res * (tota[u][e] + fabsf(x[e])) <= 0x1.0p-10f * fabsf(t[e]))) {
                    float hi, lo;
                    exact_resid<CB16>(A, K, it, ev[u] + e, x[e], hi, lo);
                    set_half(pk, e, bf16_of_pair(hi, lo));
                }
            }
            store_bf16x8(resid, ev[u], pk);
        }
    }
}

// Compensated path over UV aligned vectors (any fp32 prediction or hidden state).
template <int K, bool CB16, int UV>
__device__ __forceinline__ void vec_precise(const ExtrapArgs& A, int it, const long long (&ev)[UV]) {
    const int nb = A.nb[it];
    const int first = A.first[it];
    void* resid = A.resid[it];
    float tp[UV][8], tc[UV][8];
#pragma unroll
    for (int u = 0; u < UV; ++u)
#pragma unroll
        for (int e = 0; e < 8; ++e) tp[u][e] = tc[u][e] = 0.0f;

    for (int m = 0; m < nb; ++m) {
        const long long moff = A.m_off[first + m];
        void* out = A.m_out[first + m];
        uint4 raw[UV][K][CB16 ? 1 : 2];
        load_member<K, CB16, UV>(A, moff, ev, raw);
#pragma unroll
        for (int u = 0; u < UV; ++u) {
            float p[8], c[8];
#pragma unroll
            for (int e = 0; e < 8; ++e) p[e] = c[e] = 0.0f;
#pragma unroll
            for (int j = 0; j < K; ++j) {
                float f[8];
                unpack<CB16>(raw[u][j], f);
#pragma unroll
                for (int e = 0; e < 8; ++e) dot2_step(A.w_hi[j], A.w_lo[j], f[e], p[e], c[e]);
            }
            float hi[8], lo[8];
#pragma unroll
            for (int e = 0; e < 8; ++e) two_sum(p[e], c[e], hi[e], lo[e]);
            if (out) {
                if (A.out_bf16) {
                    uint32_t pk[4];
#pragma unroll
                    for (int i = 0; i < 4; ++i)
                        pk[i] = (uint32_t)bf16_of_pair(hi[2 * i], lo[2 * i]) |
                                ((uint32_t)bf16_of_pair(hi[2 * i + 1], lo[2 * i + 1]) << 16);
                    store_bf16x8(out, ev[u], pk);
                } else {
                    store_f32x8(out, ev[u], hi);
                }
            }
            if (resid) {
#pragma unroll
                for (int e = 0; e < 8; ++e) {
                    float q;
                    two_sum(tp[u][e], hi[e], tp[u][e], q);
                    tc[u][e] = __fadd_rn(tc[u][e], __fadd_rn(q, lo[e]));
                }
            }
        }
    }
    if (resid) {
#pragma unroll
        for (int u = 0; u < UV; ++u) {
            float x[8], hi[8], lo[8];
            load_x8(resid, A.resid_bf16, ev[u], x);
#pragma unroll
            for (int e = 0; e < 8; ++e) {
                float q;
                two_sum(tp[u][e], x[e], tp[u][e], q);
                tc[u][e] = __fadd_rn(tc[u][e], q);
                two_sum(tp[u][e], tc[u][e], hi[e], lo[e]);
            }
            if (A.resid_bf16) {
                uint32_t pk[4];
#pragma unroll
                for (int i = 0; i < 4; ++i)
                    pk[i] = (uint32_t)bf16_of_pair(hi[2 * i], lo[2 * i]) |
                            ((uint32_t)bf16_of_pair(hi[2 * i + 1], lo[2 * i + 1]) << 16);
                store_bf16x8(resid, ev[u], pk);
            } else {
                store_f32x8(resid, ev[u], hi);
            }
        }
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
            if (A.precise)
                vec_precise<K, CB16, U>(A, it, ev);
            else
                vec_fast<K, CB16, U>(A, it, ev);
        } else if (A.vec_ok[it]) {  // the ragged last tile of an aligned item
            for (int u = 0; u < U; ++u) {
                const long long v0 = e0 + ((long long)u * kThreads + threadIdx.x) * kVecElems;
                if (v0 + kVecElems <= numel) {
                    const long long ev1[1] = {v0};
                    if (A.precise)
                        vec_precise<K, CB16, 1>(A, it, ev1);
                    else
                        vec_fast<K, CB16, 1>(A, it, ev1);
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
