// Internal: the per-element arithmetic of the skipped-step kernels, shared by
// the direct-load kernel (direct_kernel.cuh) and the bulk-copy pipeline kernel
// (bulk_kernel.cuh) so that both produce identical bits.
//
// Fast path. s = sum_j w_hi[j] F_j by fp32 FMA and, alongside,
// a = sum_j |w_hi[j]| |F_j|. With u = 2^-24 the FMA chain plus the dropped low
// half of each weight give |s - P| <= (K+1) u a (1 + O(Ku)). Whenever
// (K+2) u a (1.01) <= 2^-9 |s| that error is below the smallest bf16 spacing
// next to s, so bf16(s) lies within one bf16 ulp of bf16(P). The kernels
// accumulate the bound already scaled, a' = sum_j w_guard[j] |F_j| with
// w_guard[j] = (K+2) u (1.01) 2^9 |w_hi[j]| (host-computed), so the test is
// a' <= |s|; the 1 % margin covers the extra fp32 roundings of a'.
// Elements failing the test (strong cancellation, ~1e-4..3e-3 of them) are
// recomputed from the values already loaded with Dot2 (Ogita, Rump &
// Oishi, "Accurate Sum and Dot Product", SIAM J. Sci. Comput. 26(6), 2005:
// TwoProduct by FMA plus TwoSum) with the weights as fp32 pairs hi + lo, and
// the unevaluated result pair is rounded once. fp32 results always take Dot2.
#pragma once

#include <cuda_bf16.h>

#include <type_traits>

#include "cb_device.h"

namespace cbk {
namespace {

constexpr float kU = 0x1.0p-24f;

// Plain 16-byte global load of history values (direct-load kernel). The
// streaming form (ld.global.nc with L1::no_allocate) measured slower on GB300:
// the FLUX skipped step took 2159 us with it and 1940 us without.
__device__ __forceinline__ uint4 ld_v4(const unsigned char* p) {
    uint4 v;
    asm("ld.global.v4.u32 {%0,%1,%2,%3}, [%4];" : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "l"(p));
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

template <bool CB16>
__device__ __forceinline__ void unpack(const uint4 (&r)[CB16 ? 1 : 2], float (&f)[8]) {
    if constexpr (CB16)
        unpack_bf16x8(r[0], f);
    else
        unpack_f32x8(r[0], r[CB16 ? 0 : 1], f);
}

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
    __nv_bfloat162 h = __floats2bfloat162_rn(lo, hi);  // RNE; .x is the low half
    return *reinterpret_cast<uint32_t*>(&h);
}

__device__ __forceinline__ uint16_t bf16_bits(float x) { return __bfloat16_as_ushort(__float2bfloat16_rn(x)); }

// ---- error-free transformations (explicitly rounded operations, never contracted)
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

// Start of history entry j of the member at byte offset moff.
__device__ __forceinline__ const unsigned char* hist_ptr(const ExtrapArgs& A, int j, long long moff) {
    return reinterpret_cast<const unsigned char*>(A.hist_base + (unsigned long long)A.slot_off[j] +
                                                  (unsigned long long)moff);
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

// Full-step epilogue: element e of a source converted to the output type (bit
// copy for equal types, exact widening, round-to-nearest-even narrowing).
template <bool CB16>
__device__ __forceinline__ void copy_elem(void* out, bool out_bf16, const unsigned char* src, long long e) {
    if constexpr (CB16) {
        const uint16_t h = reinterpret_cast<const uint16_t*>(src)[e];
        if (out_bf16)
            reinterpret_cast<uint16_t*>(out)[e] = h;
        else
            reinterpret_cast<uint32_t*>(out)[e] = (uint32_t)h << 16;
    } else {
        const float f = reinterpret_cast<const float*>(src)[e];
        if (out_bf16)
            reinterpret_cast<uint16_t*>(out)[e] = bf16_bits(f);
        else
            reinterpret_cast<float*>(out)[e] = f;
    }
}

// Gate of member mi (item it) at element e: g[b * hidden + h] for element
// e = (b * tokens + token) * hidden + h; 1 when the member has no gate.
__device__ __forceinline__ float gate_at(const ExtrapArgs& A, int mi, int it, long long e) {
    const void* g = A.m_gate[mi];
    if (!g) return 1.0f;
    const unsigned long long row = A.i_row[it], H = A.i_hidden[it], ue = (unsigned long long)e;
    return load_elem(g, A.gate_bf16, (long long)(ue / row * H + ue % H));
}

// Exact product g * (h + l) added to the unevaluated sum tp + tc.
__device__ __forceinline__ void add_gated_pair(float g, float h, float l, float& tp, float& tc) {
    const float gh = __fmul_rn(g, h);
    const float gr = __fmaf_rn(g, h, -gh);  // exact: g*h - gh
    float q;
    two_sum(tp, gh, tp, q);
    tc = __fadd_rn(tc, __fadd_rn(q, gr));
    tc = __fmaf_rn(g, l, tc);
}

// Compensated value of member tensor (byte offset moff) at element e.
template <bool CB16>
__device__ __noinline__ void exact_member(const ExtrapArgs& A, int K, long long moff, long long e, float& hi,
                                          float& lo) {
    float p = 0.0f, c = 0.0f;
    for (int j = 0; j < K; ++j) {
        const float f = load_cache_elem<CB16>(hist_ptr(A, j, moff), e);
        dot2_step(A.w_hi[j], A.w_lo[j], f, p, c);
    }
    two_sum(p, c, hi, lo);
}

// Compensated hidden-state update of item `it` at element e: x + sum_b P_b.
template <bool CB16>
__device__ __noinline__ void exact_resid(const ExtrapArgs& A, int K, int it, long long e, float x, float& hi,
                                         float& lo) {
    float tp = x, tc = 0.0f;
    const int first = A.first[it];
    for (int m = 0; m < A.nb[it]; ++m) {
        float h, l, q;
        exact_member<CB16>(A, K, A.m_off[first + m], e, h, l);
        if (A.m_gate[first + m]) {
            add_gated_pair(gate_at(A, first + m, it, e), h, l, tp, tc);
        } else {
            two_sum(tp, h, tp, q);
            tc = __fadd_rn(tc, __fadd_rn(q, l));
        }
    }
    two_sum(tp, tc, hi, lo);
}

// One element of item `it` through the compensated path, every member and the
// hidden state (misaligned items and ragged tails).
template <bool CB16>
__device__ __noinline__ void scalar_element(const ExtrapArgs& A, int K, int it, long long e) {
    const int first = A.first[it];
    void* resid = A.resid[it];
    float tp = 0.0f, tc = 0.0f;
    for (int m = 0; m < A.nb[it]; ++m) {
        float hi, lo, q;
        exact_member<CB16>(A, K, A.m_off[first + m], e, hi, lo);
        void* out = A.m_out[first + m];
        if (out && A.copy_out)
            copy_elem<CB16>(out, A.out_bf16, hist_ptr(A, 0, A.m_off[first + m]), e);
        else if (out)
            store_pair(out, A.out_bf16, e, hi, lo);
        if (A.m_gate[first + m]) {
            add_gated_pair(gate_at(A, first + m, it, e), hi, lo, tp, tc);
        } else {
            two_sum(tp, hi, tp, q);
            tc = __fadd_rn(tc, __fadd_rn(q, lo));
        }
    }
    if (resid) {
        float q, hi, lo;
        two_sum(tp, load_elem(resid, A.resid_bf16, e), tp, q);
        tc = __fadd_rn(tc, q);
        two_sum(tp, tc, hi, lo);
        store_pair(resid, A.resid_bf16, e, hi, lo);
    }
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

// Running sums of one item across its members (the fused hidden-state update):
// fast path x = sum_b s_b, y = sum_b a_b; compensated path x + y is the
// unevaluated sum (running value and its error).
template <int UV>
struct Acc {
    float x[UV][8];
    float y[UV][8];
    __device__ __forceinline__ void zero() {
#pragma unroll
        for (int u = 0; u < UV; ++u)
#pragma unroll
            for (int e = 0; e < 8; ++e) x[u][e] = y[u][e] = 0.0f;
    }
};

template <int K, bool CB16, int UV>
using RawVecs = uint4[UV][K][CB16 ? 1 : 2];

// Full-step epilogue: the 8 source values of vector (raw) written to out at
// element e in the output type (see copy_elem).
template <bool CB16>
__device__ __forceinline__ void copy_vec(void* out, bool out_bf16, long long e, const uint4 (&r)[CB16 ? 1 : 2]) {
    if constexpr (CB16) {
        if (out_bf16) {
            *reinterpret_cast<uint4*>(reinterpret_cast<uint16_t*>(out) + e) = r[0];
        } else {
            const uint4 v = r[0];
            uint4* q = reinterpret_cast<uint4*>(reinterpret_cast<float*>(out) + e);
            q[0] = make_uint4(v.x << 16, v.x & 0xFFFF0000u, v.y << 16, v.y & 0xFFFF0000u);
            q[1] = make_uint4(v.z << 16, v.z & 0xFFFF0000u, v.w << 16, v.w & 0xFFFF0000u);
        }
    } else {
        const uint4 a = r[0], b = r[CB16 ? 0 : 1];
        if (out_bf16) {
            *reinterpret_cast<uint4*>(reinterpret_cast<uint16_t*>(out) + e) = make_uint4(
                pack_bf16x2(__uint_as_float(a.x), __uint_as_float(a.y)), pack_bf16x2(__uint_as_float(a.z), __uint_as_float(a.w)),
                pack_bf16x2(__uint_as_float(b.x), __uint_as_float(b.y)), pack_bf16x2(__uint_as_float(b.z), __uint_as_float(b.w)));
        } else {
            uint4* q = reinterpret_cast<uint4*>(reinterpret_cast<float*>(out) + e);
            q[0] = a;
            q[1] = b;
        }
    }
}

// Output pointer handed to member_fast / member_precise for member mi: in the
// full-step epilogue the sources are written out converted here and no
// prediction is stored (null); otherwise the member's prediction output.
template <int K, bool CB16, int UV>
__device__ __forceinline__ void* member_out(const ExtrapArgs& A, int mi, const long long (&ev)[UV],
                                            const RawVecs<K, CB16, UV>& raw) {
    void* out = A.m_out[mi];
    if (!A.copy_out) return out;
    if (out)
#pragma unroll
        for (int u = 0; u < UV; ++u) copy_vec<CB16>(out, A.out_bf16, ev[u], raw[u][0]);
    return nullptr;
}

// Gate source of an ungated accumulation (never called).
struct NoGate {
    __device__ void operator()(int, float (&)[8]) const {}
};

// Placeholder for "no recompute functor" (never called).
struct NoExact {
    __device__ void operator()(int, int, float&, float&) const {}
};

// Dot2 value of element e of vector u from its K history values as loaded
// (registers or shared memory); used where the fast path's guard fails.
template <int K, bool CB16, int UV>
__device__ __forceinline__ void exact_from_raw(const ExtrapArgs& A, const RawVecs<K, CB16, UV>& raw, int u, int e,
                                               float& hi, float& lo) {
    float p = 0.0f, c = 0.0f;
#pragma unroll
    for (int j = 0; j < K; ++j) {
        float f[8];
        unpack<CB16>(raw[u][j], f);
        float fe = f[0];
#pragma unroll
        for (int i = 1; i < 8; ++i) fe = (e == i) ? f[i] : fe;
        dot2_step(A.w_hi[j], A.w_lo[j], fe, p, c);
    }
    two_sum(p, c, hi, lo);
}

// Fast-path guard: with |s - P| <= (K+1) u a (1 + O(Ku)), the test
// (K+2) u a (1.01) <= 2^-9 |s| keeps the interval between s and P shorter than
// the smallest bf16 spacing next to s (2^-8 |s| in s's binade, 2^-9 |s| below
// it), so it holds at most one rounding midpoint and bf16(s) is within one ulp
// of bf16(P). With the scaled bound a' (see above) the test is a' <= |s|.
__device__ __forceinline__ bool guard_ok(float a_scaled, float s) { return a_scaled <= fabsf(s); }

// s0, s1 += w * (f0, f1): one paired fp32 FMA, each lane rounded like fmaf.
__device__ __forceinline__ void fma_pair(float w, float f0, float f1, float& s0, float& s1) {
    const float2 r = __ffma2_rn(make_float2(w, w), make_float2(f0, f1), make_float2(s0, s1));
    s0 = r.x;
    s1 = r.y;
}

// Fast path for one member over UV aligned 8-element vectors already loaded
// into registers: bf16 prediction (if out) and accumulation into acc. The
// rare guarded elements are recomputed by exact(u, e, hi, lo) when given
// (e.g. from shared memory), else from the loaded values (FROM_RAW: no memory
// latency, but the values stay live and cost registers) or re-read from
// global memory (member byte offset moff).
// GATED: gate(u, g) supplies the 8 gate values of vector u when it is
// accumulated (late, so that they are not live beside the history values).
template <int K, bool CB16, int UV, bool FROM_RAW, bool GATED = false, typename Gate = NoGate,
          typename Exact = NoExact>
__device__ __forceinline__ void member_fast(const ExtrapArgs& A, long long moff, void* out,
                                            const long long (&ev)[UV], const RawVecs<K, CB16, UV>& raw,
                                            bool accumulate, Acc<UV>& acc, Gate gate = {}, Exact exact = {}) {
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
            for (int e = 0; e < 8; e += 2) fma_pair(A.w_hi[j], f[e], f[e + 1], s[e], s[e + 1]);
#pragma unroll
            for (int e = 0; e < 8; ++e) a[e] = fmaf(A.w_guard[j], fabsf(f[e]), a[e]);
        }
        if (out) {
            uint32_t pk[4];
#pragma unroll
            for (int i = 0; i < 4; ++i) pk[i] = pack_bf16x2(s[2 * i], s[2 * i + 1]);
            unsigned bad = 0;
#pragma unroll
            for (int e = 0; e < 8; ++e) bad |= guard_ok(a[e], s[e]) ? 0u : (1u << e);
            store_bf16x8(out, ev[u], pk);
            // rare: the failing elements get their Dot2 value, stored by this
            // thread over the fast-path bf16 it has just written (the vector is
            // dead by then, so the loop keeps nothing of the fast path live)
            while (bad) {
                const int e = __ffs(bad) - 1;
                bad &= bad - 1;
                float hi, lo;
                if constexpr (!std::is_same_v<Exact, NoExact>)
                    exact(u, e, hi, lo);
                else if constexpr (FROM_RAW)
                    exact_from_raw<K, CB16, UV>(A, raw, u, e, hi, lo);
                else
                    exact_member<CB16>(A, K, moff, ev[u] + e, hi, lo);
                reinterpret_cast<uint16_t*>(out)[ev[u] + e] = bf16_of_pair(hi, lo);
            }
        }
        if (accumulate) {
            float g[8];
            if constexpr (GATED) gate(u, g);
#pragma unroll
            for (int e = 0; e < 8; ++e) {
                if constexpr (GATED) {  // x + g * s: one rounding, bound |g| a'
                    acc.x[u][e] = fmaf(g[e], s[e], acc.x[u][e]);
                    acc.y[u][e] = fmaf(fabsf(g[e]), a[e], acc.y[u][e]);
                } else {
                    acc.x[u][e] += s[e];
                    acc.y[u][e] += a[e];
                }
            }
        }
    }
}

// Full-step epilogue (a one-entry history of weight 1): member features f,
// taken exactly, added into the hidden-state sums, acc.x += g f and the
// unscaled bound acc.y += |g f| (g = 1 without gates). resid_fast scales the
// bound with yscale = w_guard[0] = 3 u (1.01) 2^9, the scaled bound the general
// path would have accumulated for K = 1.
template <int K, bool CB16, int UV, bool GATED = false, typename Gate = NoGate>
__device__ __forceinline__ void member_one(const RawVecs<K, CB16, UV>& raw, Acc<UV>& acc, Gate gate = {}) {
    static_assert(K == 1, "a one-entry history");
#pragma unroll
    for (int u = 0; u < UV; ++u) {
        float g[8];
        if constexpr (GATED) gate(u, g);  // first: each feature is then unpacked as it is used
        const uint32_t w[8] = {raw[u][0][0].x, raw[u][0][0].y, raw[u][0][0].z, raw[u][0][0].w,
                               raw[u][0][CB16 ? 0 : 1].x, raw[u][0][CB16 ? 0 : 1].y, raw[u][0][CB16 ? 0 : 1].z,
                               raw[u][0][CB16 ? 0 : 1].w};
#pragma unroll
        for (int e = 0; e < 8; ++e) {
            const float f = CB16 ? __uint_as_float((e & 1) ? (w[e >> 1] & 0xFFFF0000u) : (w[e >> 1] << 16))
                                 : __uint_as_float(w[e]);
            if constexpr (GATED) {
                acc.x[u][e] = fmaf(g[e], f, acc.x[u][e]);
                acc.y[u][e] = fmaf(fabsf(g[e]), fabsf(f), acc.y[u][e]);
            } else {
                acc.x[u][e] += f;
                acc.y[u][e] += fabsf(f);
            }
        }
    }
}

// Fast path: hidden state <- bf16(x + sum_b s_b), guarded like the members.
// xload(u, x) supplies the 8 hidden-state values of vector u (global or shared
// memory); exact(u, e, x_e, hi, lo) recomputes one guarded element with Dot2.
// yscale: factor that turns acc.y into the scaled bound (1 when the members
// accumulated scaled bounds; w_guard[0] after member_one's unscaled sums).
template <int K, int UV, typename XLoad, typename Exact>
__device__ __forceinline__ void resid_fast(const ExtrapArgs& A, int it, const long long (&ev)[UV],
                                           const Acc<UV>& acc, void* resid, XLoad xload, Exact exact,
                                           float yscale = 1.0f) {
    // the test g_res (sum_b a_b + |x|) <= 2^-9 |t|, g_res = (K + nb + 3) u 1.01,
    // on the scaled bounds acc.y = (K+2) u 1.01 2^9 sum_b a_b:
    // q acc.y + r |x| <= |t| with q = (K + nb + 3) / (K + 2), r = g_res 2^9
    const float kn = (float)(K + A.nb[it] + 3);
    const float q = kn * (1.0f / (float)(K + 2)) * 1.0000005f * yscale;  // rounded up past fp32 error
    const float r = kn * (kU * 1.01f * 512.0f);
#pragma unroll
    for (int u = 0; u < UV; ++u) {
        float x[8], t[8];
        uint32_t pk[4];
        xload(u, x);
#pragma unroll
        for (int e = 0; e < 8; ++e) t[e] = acc.x[u][e] + x[e];
#pragma unroll
        for (int i = 0; i < 4; ++i) pk[i] = pack_bf16x2(t[2 * i], t[2 * i + 1]);
        float b[8];
        bool pass = true;
#pragma unroll
        for (int e = 0; e < 8; ++e) {
            b[e] = fmaf(r, fabsf(x[e]), q * acc.y[u][e]);
            pass = pass && guard_ok(b[e], t[e]);
        }
        unsigned bad = 0;
        if (!pass)
#pragma unroll
            for (int e = 0; e < 8; ++e) bad |= guard_ok(b[e], t[e]) ? 0u : (1u << e);
        store_bf16x8(resid, ev[u], pk);
        // rare: Dot2 values stored over the fast-path bf16 just written
        while (bad) {
            const int e = __ffs(bad) - 1;
            bad &= bad - 1;
            float xe = x[0];
#pragma unroll
            for (int i = 1; i < 8; ++i) xe = (e == i) ? x[i] : xe;
            float hi, lo;
            exact(u, e, xe, hi, lo);
            reinterpret_cast<uint16_t*>(resid)[ev[u] + e] = bf16_of_pair(hi, lo);
        }
    }
}

// Compensated path for one member (any fp32 prediction or hidden state).
template <int K, bool CB16, int UV, bool GATED = false, typename Gate = NoGate>
__device__ __forceinline__ void member_precise(const ExtrapArgs& A, void* out, const long long (&ev)[UV],
                                               const RawVecs<K, CB16, UV>& raw, bool accumulate,
                                               Acc<UV>& acc, Gate gate = {}) {
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
        if (accumulate) {
            float g[8];
            if constexpr (GATED) gate(u, g);
#pragma unroll
            for (int e = 0; e < 8; ++e) {
                if constexpr (GATED) {
                    add_gated_pair(g[e], hi[e], lo[e], acc.x[u][e], acc.y[u][e]);
                } else {
                    float q;
                    two_sum(acc.x[u][e], hi[e], acc.x[u][e], q);
                    acc.y[u][e] = __fadd_rn(acc.y[u][e], __fadd_rn(q, lo[e]));
                }
            }
        }
    }
}

template <int UV, typename XLoad>
__device__ __forceinline__ void resid_precise(const ExtrapArgs& A, const long long (&ev)[UV], Acc<UV>& acc,
                                              void* resid, XLoad xload) {
#pragma unroll
    for (int u = 0; u < UV; ++u) {
        float x[8], hi[8], lo[8];
        xload(u, x);
#pragma unroll
        for (int e = 0; e < 8; ++e) {
            float q;
            two_sum(acc.x[u][e], x[e], acc.x[u][e], q);
            acc.y[u][e] = __fadd_rn(acc.y[u][e], q);
            two_sum(acc.x[u][e], acc.y[u][e], hi[e], lo[e]);
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

// n / d for n, d < 2^32 from M = ceil(2^64 / d) (M = 0 encodes d = 1):
// n M / 2^64 = n / d + n delta / (d 2^64) with 0 <= delta < d, and the excess
// n delta / (d 2^64) < 2^-32 < 1 / d cannot carry frac(n / d) <= (d - 1) / d
// past the next integer (division by invariant integers, after Granlund &
// Montgomery, PLDI 1994).
__device__ __forceinline__ unsigned div_magic(unsigned n, unsigned long long M) {
    return M ? (unsigned)__umul64hi((unsigned long long)n, M) : n;
}

// Gate offsets b * hidden + h of UV vectors of a tile starting at element e0
// (32-bit arithmetic: gated tensors have fewer than 2^32 elements); with
// `relative`, b counts from the tile's first batch (the staged gate rows).
// Rows of tokens * hidden are multiples of hidden, so h = e mod hidden.
template <int UV>
__device__ __forceinline__ void gate_offsets(const ExtrapArgs& A, int it, long long e0,
                                             const long long (&ev)[UV], unsigned (&gi)[UV], bool relative = false) {
    const unsigned row = A.i_row[it], H = A.i_hidden[it], ue0 = (unsigned)e0;
    if (row == 0 || H == 0) {  // no shape: no gate
#pragma unroll
        for (int u = 0; u < UV; ++u) gi[u] = 0;
        return;
    }
    const unsigned q0 = div_magic(ue0, A.i_row_magic[it]), r0 = ue0 - q0 * row;
#pragma unroll
    for (int u = 0; u < UV; ++u) {
        unsigned r = r0 + (unsigned)(ev[u] - e0), b = relative ? 0u : q0;
        while (r >= row) {  // a tile spans few rows
            r -= row;
            ++b;
        }
        const unsigned h = r - div_magic(r, A.i_hidden_magic[it]) * H;
        gi[u] = b * H + h;
    }
}

// The 8 gate values of member mi for each of UV vectors (1 without a gate).
template <int UV>
__device__ __forceinline__ void load_gates(const ExtrapArgs& A, int mi, const unsigned (&gi)[UV], float (&g)[UV][8]) {
    const void* gp = A.m_gate[mi];
#pragma unroll
    for (int u = 0; u < UV; ++u) {
        if (gp)
            load_x8(gp, A.gate_bf16, (long long)gi[u], g[u]);
        else
#pragma unroll
            for (int e = 0; e < 8; ++e) g[u][e] = 1.0f;
    }
}

}  // namespace
}  // namespace cbk
