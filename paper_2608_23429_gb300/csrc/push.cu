// Full-step cache write (Sec. 3.3: the features of a full computation are
// stored in the history buffer H; Alg. 1, full-computation branch). One
// grouped launch writes every branch tensor of every block into the ring slot
// being replaced: a bit copy for bf16 -> bf16 and fp32 -> fp32, an exact
// widening for bf16 -> fp32, and round-to-nearest-even for fp32 -> bf16.
// Like the skipped-step kernel it is a persistent grid over 4096-element
// tiles, each thread moving two 8-element vectors with both loads issued first.
#include <cuda_bf16.h>

#include "cb_device.h"

namespace cbk {
namespace {

// Plain 16-byte global load. The streaming form (ld.global.nc with
// L1::no_allocate) measured 4.5 % slower on a 1:1 copy of the FLUX slot on
// GB300 (663 against 635 us for 2 x 2.15 GB at 4 CTAs per SM).
__device__ __forceinline__ uint4 ld_v4(const void* p) {
    uint4 v;
    asm("ld.global.v4.u32 {%0,%1,%2,%3}, [%4];" : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "l"(p));
    return v;
}

__device__ __forceinline__ uint32_t pack_bf16x2(uint32_t lo_bits, uint32_t hi_bits) {
    __nv_bfloat162 h = __floats2bfloat162_rn(__uint_as_float(lo_bits), __uint_as_float(hi_bits));
    return *reinterpret_cast<uint32_t*>(&h);
}

template <bool SB>
struct Raw {
    uint4 w[SB ? 1 : 2];  // 8 source elements
};

template <bool SB>
__device__ __forceinline__ Raw<SB> load8(const void* src, long long e) {
    Raw<SB> r;
    if constexpr (SB) {
        r.w[0] = ld_v4(reinterpret_cast<const uint16_t*>(src) + e);
    } else {
        const float* p = reinterpret_cast<const float*>(src) + e;
        r.w[0] = ld_v4(p);
        r.w[SB ? 0 : 1] = ld_v4(p + 4);
    }
    return r;
}

template <bool SB, bool DB>
__device__ __forceinline__ void store8(unsigned char* dst, long long e, const Raw<SB>& r) {
    if constexpr (SB && DB) {
        *reinterpret_cast<uint4*>(reinterpret_cast<uint16_t*>(dst) + e) = r.w[0];
    } else if constexpr (!SB && DB) {
        const uint4 a = r.w[0], b = r.w[SB ? 0 : 1];
        *reinterpret_cast<uint4*>(reinterpret_cast<uint16_t*>(dst) + e) =
            make_uint4(pack_bf16x2(a.x, a.y), pack_bf16x2(a.z, a.w), pack_bf16x2(b.x, b.y), pack_bf16x2(b.z, b.w));
    } else if constexpr (SB && !DB) {
        const uint4 v = r.w[0];
        uint4* q = reinterpret_cast<uint4*>(reinterpret_cast<float*>(dst) + e);
        q[0] = make_uint4(v.x << 16, v.x & 0xFFFF0000u, v.y << 16, v.y & 0xFFFF0000u);
        q[1] = make_uint4(v.z << 16, v.z & 0xFFFF0000u, v.w << 16, v.w & 0xFFFF0000u);
    } else {
        uint4* q = reinterpret_cast<uint4*>(reinterpret_cast<float*>(dst) + e);
        q[0] = r.w[0];
        q[1] = r.w[SB ? 0 : 1];
    }
}

template <bool SB, bool DB>
__device__ __forceinline__ void copy1(unsigned char* dst, const void* src, long long e) {
    if constexpr (SB && DB) {
        reinterpret_cast<uint16_t*>(dst)[e] = reinterpret_cast<const uint16_t*>(src)[e];
    } else if constexpr (!SB && DB) {
        reinterpret_cast<__nv_bfloat16*>(dst)[e] = __float2bfloat16_rn(reinterpret_cast<const float*>(src)[e]);
    } else if constexpr (SB && !DB) {
        reinterpret_cast<uint32_t*>(dst)[e] = (uint32_t)(reinterpret_cast<const uint16_t*>(src)[e]) << 16;
    } else {
        reinterpret_cast<uint32_t*>(dst)[e] = reinterpret_cast<const uint32_t*>(src)[e];
    }
}

template <bool SB, bool DB>
__global__ void __launch_bounds__(kThreads) push_kernel(const __grid_constant__ PushArgs A) {
    constexpr long long TE = push_tile_elems;
    int it = 0;
    for (int tile = blockIdx.x; tile < A.tiles_total; tile += gridDim.x) {
        while (tile >= A.tile_begin[it + 1]) ++it;
        const long long numel = A.numel[it];
        const long long e0 = (long long)(tile - A.tile_begin[it]) * TE;
        unsigned char* dst = A.slot + A.off[it];
        const void* src = A.src[it];
        if (A.vec_ok[it] && e0 + TE <= numel) {
            const long long ea = e0 + (long long)threadIdx.x * kVecElems;
            const long long eb = ea + (long long)kThreads * kVecElems;
            const Raw<SB> ra = load8<SB>(src, ea);
            const Raw<SB> rb = load8<SB>(src, eb);
            store8<SB, DB>(dst, ea, ra);
            store8<SB, DB>(dst, eb, rb);
        } else {
            const long long end = e0 + TE < numel ? e0 + TE : numel;
            for (long long e = e0 + threadIdx.x; e < end; e += kThreads) copy1<SB, DB>(dst, src, e);
        }
    }
}

template <bool SB, bool DB>
cudaError_t launch_t(const PushArgs& a, int grid, cudaStream_t s) {
    push_kernel<SB, DB><<<grid, kThreads, 0, s>>>(a);
    return cudaGetLastError();
}

template <bool SB, bool DB>
cudaError_t occ_t(int* blocks) {
    return cudaOccupancyMaxActiveBlocksPerMultiprocessor(blocks, push_kernel<SB, DB>, kThreads, 0);
}

}  // namespace

cudaError_t launch_push(const PushArgs& a, bool src_bf16, bool dst_bf16, int grid, cudaStream_t s) {
    if (src_bf16) return dst_bf16 ? launch_t<true, true>(a, grid, s) : launch_t<true, false>(a, grid, s);
    return dst_bf16 ? launch_t<false, true>(a, grid, s) : launch_t<false, false>(a, grid, s);
}

cudaError_t push_blocks_per_sm(bool src_bf16, bool dst_bf16, int* blocks) {
    if (src_bf16) return dst_bf16 ? occ_t<true, true>(blocks) : occ_t<true, false>(blocks);
    return dst_bf16 ? occ_t<false, true>(blocks) : occ_t<false, false>(blocks);
}

}  // namespace cbk
