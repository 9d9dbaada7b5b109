// Full-step epilogue kernel (cb_cache_push_residual; Sec. 3.3 / Alg. 1,
// full-computation branch, plus the block residual of Sec. 3.1): every branch
// output is written into the ring slot (bit copy, exact widening or RNE
// narrowing, as the cache write) and, for each residual group,
//     x <- round(x + sum_b g_b f_b)
// with the features taken un-rounded.
//
// A one-entry history of weight 1 needs no weighted sum, and the pattern is
// one byte out per byte in, that of a plain copy. So the kernel is shaped like
// the cache write: a persistent grid of three 256-thread CTAs per SM over
// 2048-element tiles, each thread loading one 8-element vector of every
// member's features and of the hidden state (plain 16-byte loads, all issued
// before any arithmetic), then storing the slot vectors and the new hidden
// state. The arithmetic is the skipped-step kernels' (cb_math.cuh), with the
// same choices per case as the direct-load kernel, so the kernels write
// identical bits (the bulk kernel's ragged last tiles, computed by the
// compensated path throughout, aside).
//
// Each thread has (members + 1) loads in flight, so the kernel streams well
// only when groups are large: the host runs it for ungated bf16 features when
// every tensor belongs to a residual group of three or more branches (GB300,
// PixArt-Sigma 1024^2, groups of 3: 96.1 % of the copy peak against 91.4 % for
// the bulk pipeline; FLUX.1-dev, groups of 1 and 2: 82.4 % against 93.9 %).
#include "direct_kernel.cuh"

namespace cbk {
namespace {

constexpr int kEpilogueCtasPerSm = 3;
constexpr int kEpilogueMaxMembers = 4;  // CB_MAX_BRANCHES branch tensors per residual group
static_assert(epilogue_tile_elems == (long long)kThreads * kVecElems, "one vector per thread and tile");

// One 8-element vector (element ev[0]) of item `it` through every member and
// the hidden state.
template <bool CB16, bool GATED>
__device__ __forceinline__ void epilogue_vector(const ExtrapArgs& A, int it, const long long (&ev)[1]) {
    const int nb = A.nb[it];
    const int first = A.first[it];
    void* resid = A.resid[it];
    // loads first: every member's features and the bf16 hidden state
    RawVecs<1, CB16, 1> raw[kEpilogueMaxMembers];
#pragma unroll
    for (int m = 0; m < kEpilogueMaxMembers; ++m)
        if (m < nb) load_member<1, CB16, 1>(A, A.m_off[first + m], ev, raw[m]);
    const bool x16 = resid != nullptr && A.resid_bf16;
    uint4 xr = make_uint4(0u, 0u, 0u, 0u);
    if (x16) xr = ld_v4(reinterpret_cast<const unsigned char*>(resid) + ev[0] * 2);
    unsigned gi[1] = {0u};
    if constexpr (GATED) {  // items without shapes carry no gate
        if (resid && A.i_hidden[it] != 0) gate_offsets<1>(A, it, ev[0], ev, gi);
    }
    Acc<1> acc;
    acc.zero();
#pragma unroll
    for (int m = 0; m < kEpilogueMaxMembers; ++m) {
        if (m >= nb) break;
        member_out<1, CB16, 1>(A, first + m, ev, raw[m]);  // the slot write
        if (!resid) continue;
        const void* gp = GATED ? A.m_gate[first + m] : nullptr;
        auto gate = [&](int, float (&gv)[8]) {
            if (gp)
                load_x8(gp, A.gate_bf16, (long long)gi[0], gv);
            else
#pragma unroll
                for (int e = 0; e < 8; ++e) gv[e] = 1.0f;
        };
        if (A.precise)
            member_precise<1, CB16, 1, GATED>(A, nullptr, ev, raw[m], true, acc, gate);
        else if constexpr (CB16)  // bf16 features: exact, no weighted sum
            member_one<1, CB16, 1, GATED>(raw[m], acc, gate);
        else
            member_fast<1, CB16, 1, false, GATED>(A, A.m_off[first + m], nullptr, ev, raw[m], true, acc, gate);
    }
    if (!resid) return;
    auto xload = [&](int, float (&x)[8]) {
        if (x16)
            unpack_bf16x8(xr, x);
        else
            load_x8(resid, false, ev[0], x);
    };
    if (A.precise) {
        resid_precise<1>(A, ev, acc, resid, xload);
    } else {
        resid_fast<1, 1>(
            A, it, ev, acc, resid, xload,
            [&](int, int e, float xe, float& hi, float& lo) { exact_resid<CB16>(A, 1, it, ev[0] + e, xe, hi, lo); },
            CB16 ? A.w_guard[0] : 1.0f);
    }
}

template <bool CB16, bool GATED>
__global__ void __launch_bounds__(kThreads, kEpilogueCtasPerSm) epilogue_kernel(const __grid_constant__ ExtrapArgs A) {
    constexpr long long TE = epilogue_tile_elems;
    int it = 0;
    for (int tile = blockIdx.x; tile < A.tiles_total; tile += gridDim.x) {
        while (tile >= A.tile_begin[it + 1]) ++it;  // tiles only grow: walk forward
        const long long numel = A.numel[it];
        const long long e0 = (long long)(tile - A.tile_begin[it]) * TE;
        const long long v0 = e0 + (long long)threadIdx.x * kVecElems;
        if (A.vec_ok[it] && v0 + kVecElems <= numel) {
            const long long ev[1] = {v0};
            epilogue_vector<CB16, GATED>(A, it, ev);
        } else if (A.vec_ok[it]) {  // the end of the ragged last tile of an aligned item
            for (long long e = v0; e < numel && e < v0 + kVecElems; ++e) scalar_element<CB16>(A, 1, it, e);
        } else {  // misaligned item: element-wise, adjacent threads on adjacent elements
            const long long end = e0 + TE < numel ? e0 + TE : numel;
            for (long long e = e0 + threadIdx.x; e < end; e += kThreads) scalar_element<CB16>(A, 1, it, e);
        }
    }
}

}  // namespace

// Only the case the host runs here is instantiated: bf16 features, no gates.
cudaError_t launch_epilogue(const ExtrapArgs& a, int grid, cudaStream_t s) {
    epilogue_kernel<true, false><<<grid, kThreads, 0, s>>>(a);
    return cudaGetLastError();
}

cudaError_t epilogue_blocks_per_sm(int* blocks) {
    return cudaOccupancyMaxActiveBlocksPerMultiprocessor(blocks, epilogue_kernel<true, false>, kThreads, 0);
}

}  // namespace cbk
