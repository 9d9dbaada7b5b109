// Skipped-step kernel, bulk-copy pipeline variant (same arithmetic and bits as
// the direct kernel on whole tiles; a tensor's ragged last tile takes the
// compensated path for every element here. Sec. 3.3, Eq. for f_t; Alg. 1,
// extrapolation branch).
//
// One or two CTAs per SM (see Shape). A producer lane moves,
// for every work unit (one tile of one branch tensor), the K history chunks of
// 8 KB each from HBM into a ring of shared-memory stages with cp.async.bulk
// (the Blackwell bulk-copy engine), each stage guarded by a "full" mbarrier
// (transaction bytes) and an "empty" mbarrier (one arrival per consumer warp).
// Consumer warps read their 8-element vectors of the K chunks from shared
// memory, compute, and store from registers. With S stages of K x 8 KB (S = 5
// for K = 5) up to ~200 KB per SM stay in flight independently of the
// consumers' registers, which is what bounds the direct-load variant.
//
// Many consumer warps per scheduler hide the consumers' fixed latencies (see
// Shape for the thread map). Every consumer fences its reads of a stage
// against the async proxy before the stage goes back to the producer
// (release_stage). Two kinds of launch (GROUPED):
//   * predictions only: each stage is released as soon as it is read into
//     registers, and guarded elements are recomputed from those registers;
//   * with hidden states: stages are released after the member's arithmetic,
//     guarded elements are recomputed from shared memory (so the history
//     values die early). The producer also stages each tile's bf16 hidden
//     state (one more chunk with the group's last member) and the consumers
//     hold the group's member stages until the hidden state is written (the
//     host guarantees more stages than members, so holding cannot starve the
//     producer). With gates, each member's stage also carries the gate rows
//     of the batches its tile touches, so that no consumer waits on a global
//     load.
// The same kernel runs a full step's epilogue (cb_cache_push_residual) as a
// one-entry history of weight 1 whose member addresses are the new features;
// with copy_out the outputs (the ring slot) receive the features converted.
//
// Every wait is bounded (%globaltimer). A consumer wait that runs out in any
// lane records a code in the plan's device status word and the whole warp
// returns (a warp vote, so no lane leaves a warp that goes on to a
// __syncwarp); a producer wait that runs out stops the producer, which then
// waits, with its own limit (at least 10 ms), for the copies it has issued
// before it exits. A test option makes the producer announce the first unit's
// bytes without issuing its copies, so that the consumers' wait runs out with
// no fault and nothing in flight.
#pragma once

#include "cb_async.cuh"
#include "cb_math.cuh"

namespace cbk {
namespace {

// Thread map. With one CTA per SM, one 8-element vector per consumer thread
// and tile: 16 consumer warps for bf16 tiles (512 vectors; 17 warps cap
// registers at 96), 8 for fp32 tiles (256 vectors). Launches that carry few
// bytes per unit (most K = 1 launches, and bf16 launches with small K: see
// bulk_ctas_per_sm) pay the consumers' fixed cost per unit more often; they run two CTAs of 8
// consumer warps per SM (two independent pipelines), bf16 threads taking two
// vectors per tile. An earlier map of 8 consumer warps with two vectors each
// on one CTA left the launches with hidden states issue-bound.
template <bool CB16, int K, bool GROUPED, bool GATED>
struct Shape {
    static constexpr int ctas_per_sm = bulk_ctas_per_sm(K, CB16, GROUPED, GATED);
    static constexpr int consumer_warps = (CB16 && ctas_per_sm == 1) ? 16 : 8;
    static constexpr int consumers = consumer_warps * 32;
    static constexpr int threads = consumers + 32;  // plus the producer warp
};
constexpr int kChunkBytes = 8192;   // one history entry's share of a tile
constexpr int kBarrierBytes = 256;  // full[S] and empty[S] barriers, S <= kMaxStages
static_assert(2 * 8 * kMaxStages <= kBarrierBytes, "barrier block holds every stage's barriers");
// A consumer warp hands one stage back to the producer: every lane fences its
// shared-memory reads of the stage against the async proxy, then lane 0
// arrives on the stage's empty barrier. The refill that follows is an
// async-proxy write to the same bytes, and the mbarrier release/acquire pair
// alone does not order it after generic-proxy reads: without the fence, a
// refill landed on the start of a stage before some of a warp's loads were
// performed (half a warp's first vector took the next unit's bytes, about one
// launch in 200 on full-size PixArt shapes; none in 3000 with the fence).
__device__ __forceinline__ void release_stage(uint32_t empty_bar, int lane) {
    fence_generic_to_async();
    __syncwarp();
    if (lane == 0) mbar_arrive(empty_bar);
}

// GROUPED: some item updates a hidden state or has several members (stage
// holding, hidden-state staging); prediction-only launches compile without
// that bookkeeping. GATED (with GROUPED): the hidden state receives g_b * P_b,
// with a per-(batch, channel) gate per member.
// ONE: the full-step epilogue (copy_out with bf16 hidden states or none): a
// one-entry history of weight 1, whose member step needs no weighted sum
// (member_one); compiled apart so that each kernel carries only its own path.
template <int K, bool CB16, bool GROUPED, bool GATED, bool ONE = false>
__global__ void __launch_bounds__(Shape<CB16, K, GROUPED, GATED>::threads, Shape<CB16, K, GROUPED, GATED>::ctas_per_sm)
    extrapolate_bulk_kernel(const __grid_constant__ ExtrapArgs A) {
    static_assert(!ONE || K == 1, "the epilogue is a one-entry history");
    extern __shared__ __align__(128) unsigned char smem[];
    constexpr int NCW = Shape<CB16, K, GROUPED, GATED>::consumer_warps;
    constexpr int NCT = Shape<CB16, K, GROUPED, GATED>::consumers;
    constexpr long long TE = tile_elems(CB16);  // 8 KB per history chunk for both cache types
    constexpr int ES = CB16 ? 2 : 4;
    constexpr int NV = (int)(TE / kVecElems);     // vectors per tile: 512 (bf16) or 256 (fp32)
    constexpr int U = NV >= NCT ? NV / NCT : 1;   // vectors per consumer thread per tile
    static_assert(NV % NCT == 0 || NCT % NV == 0, "vectors spread evenly over the consumers");
    static_assert(TE * ES == kChunkBytes, "one tile of one history entry is one chunk");
    const int S = A.stages;
    const uint32_t full0 = smem_addr(smem);
    const uint32_t empty0 = full0 + 8u * (uint32_t)S;
    const uint32_t buf0 = smem_addr(smem + kBarrierBytes);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

    if (threadIdx.x == 0) {
        for (int s = 0; s < S; ++s) {
            mbar_init(full0 + 8u * s, 1);
            mbar_init(empty0 + 8u * s, NCW);
        }
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    __syncthreads();

    // the stage stays held through the member's arithmetic (see the consumers)
    constexpr bool LATE = GROUPED || (CB16 && K >= 7);
    const int C = GROUPED ? A.stage_chunks : K;
    const uint32_t stage_bytes = (uint32_t)C * kChunkBytes + (GATED ? A.stage_gate_bytes : 0u);
    if (warp == NCW) {  // ---------------------------------- producer
        if (lane != 0) return;
        int it = 0;
        unsigned u = 0;               // units issued
        uint32_t ps = 0, wraps = 0;   // stage of the next unit; times the ring has wrapped
        bool ok = true;
        for (int tile = blockIdx.x; ok && tile < A.tiles_total; tile += gridDim.x) {
            while (tile >= A.tile_begin[it + 1]) ++it;
            const long long numel = A.numel[it];
            const long long e0 = (long long)(tile - A.tile_begin[it]) * TE;
            // consumers read shared memory only for whole tiles of aligned items;
            // for the ragged last tile (or a misaligned item) the stage is
            // cycled without data and they recompute from global memory
            const bool full_tile = A.vec_ok[it] && e0 + TE <= numel;
            const uint32_t bytes = full_tile ? (uint32_t)kChunkBytes : 0u;
            const int first = A.first[it];
            const int nb = GROUPED ? A.nb[it] : 1;
            const unsigned char* resid = GROUPED ? reinterpret_cast<const unsigned char*>(A.resid[it]) : nullptr;
            // gate rows b0..b1 of the batches this tile touches (b1 <= b0 + 1:
            // the host stages gates only when a batch holds a tile or more)
            uint32_t gbytes = 0;
            size_t gsrc = 0;
            if (GATED && A.stage_gate_bytes && resid && full_tile && A.i_row[it] != 0) {
                const long long row = A.i_row[it];
                const long long b0 = e0 / row, b1 = (e0 + TE - 1) / row;
                const size_t gs = A.gate_bf16 ? 2 : 4;
                gsrc = (size_t)b0 * A.i_hidden[it] * gs;
                gbytes = (uint32_t)((b1 - b0 + 1) * A.i_hidden[it] * gs);
            }
            for (int m = 0; m < nb; ++m) {
                const uint32_t stage = ps;
                if (wraps > 0 && !mbar_wait(empty0 + 8u * stage, (wraps - 1) & 1u, A.wait_ns)) {
                    record(A.status, 2);
                    ok = false;
                    break;
                }
                ++u;
                if (++ps == (uint32_t)S) {
                    ps = 0;
                    ++wraps;
                }
                // the tile's bf16 hidden state travels with its last member
                const bool with_x = GROUPED && A.stage_x && resid && full_tile && m == nb - 1;
                const uint32_t xbytes = with_x ? (uint32_t)(TE * 2) : 0u;
                const uint32_t gb = (GATED && A.m_gate[first + m]) ? gbytes : 0u;
                mbar_expect_tx(full0 + 8u * stage, (uint32_t)K * bytes + xbytes + gb);
                if (A.withhold_first && u == 1) continue;
                const uint32_t dst = buf0 + stage * stage_bytes;
                if (bytes) {
#pragma unroll
                    for (int j = 0; j < K; ++j)
                        bulk_g2s(dst + j * (uint32_t)kChunkBytes, hist_ptr(A, j, A.m_off[first + m]) + e0 * ES, bytes,
                                 full0 + 8u * stage);
                }
                if (xbytes) bulk_g2s(dst + K * (uint32_t)kChunkBytes, resid + e0 * 2, xbytes, full0 + 8u * stage);
                if (gbytes && A.m_gate[first + m])
                    bulk_g2s(dst + C * (uint32_t)kChunkBytes,
                             reinterpret_cast<const unsigned char*>(A.m_gate[first + m]) + gsrc, gbytes,
                             full0 + 8u * stage);
            }
        }
        // never leave while copies into this CTA's shared memory are in flight:
        // wait for every unit still in the ring; after one wait runs out (a unit
        // whose copies were never issued) the others get the short limit
        unsigned long long drain_ns = A.wait_ns > kMinDrainNs ? A.wait_ns : kMinDrainNs;
        bool drained = true;
        for (unsigned q = u > (unsigned)S ? u - S : 0; q < u; ++q)
            if (!mbar_wait(full0 + 8u * (q % S), (q / S) & 1u, drain_ns)) {
                drained = false;
                drain_ns = kMinDrainNs;
            }
        if (!drained) record(A.status, 4);
        return;
    }

    // ------------------------------------------------------------ consumers
    const int c = threadIdx.x;
    const unsigned char* stages = smem + kBarrierBytes;
    auto chunk = [&](uint32_t stage, int j) { return stages + stage * stage_bytes + (size_t)j * kChunkBytes; };
    auto gate_stage = [&](uint32_t stage) -> const void* { return stages + stage * stage_bytes + (size_t)C * kChunkBytes; };
    int it = 0;
    uint32_t cs = 0, cph = 0;  // stage of the next unit to consume and its phase parity
    for (int tile = blockIdx.x; tile < A.tiles_total; tile += gridDim.x) {
        while (tile >= A.tile_begin[it + 1]) ++it;
        const long long numel = A.numel[it];
        const long long e0 = (long long)(tile - A.tile_begin[it]) * TE;
        const int nb = GROUPED ? A.nb[it] : 1;
        const int first = A.first[it];
        void* resid = GROUPED ? A.resid[it] : nullptr;
        // whole aligned tiles come from shared memory; the ragged last tile of a
        // tensor and misaligned items take the compensated scalar path
        const bool full_tile = A.vec_ok[it] && e0 + TE <= numel;
        // with a hidden state, every member's stage stays held until the hidden
        // state is written, so that its guarded elements can be recomputed
        const bool hold = GROUPED && full_tile && resid != nullptr;
        const bool mine = NV >= NCT || c < NV;  // fp32 tiles have fewer vectors than consumers
        // stage of member m of this tile (nb < S: one wrap at most)
        const uint32_t s0 = cs;
        auto stage_of = [&](int m) { return s0 + m < (uint32_t)S ? s0 + m : s0 + m - (uint32_t)S; };
        long long ev[U];
#pragma unroll
        for (int v = 0; v < U; ++v) ev[v] = e0 + ((long long)v * NCT + c) * kVecElems;
        // gate offsets of this thread's vectors, relative to the gate rows the
        // producer staged (or absolute, when gates stay in global memory)
        unsigned gi[U];
        if constexpr (GATED) {
            if (hold && A.i_row[it] != 0)  // items without a shape carry no gate
                gate_offsets<U>(A, it, e0, ev, gi, A.stage_gate_bytes != 0);
        }
        Acc<U> acc;
        acc.zero();
        for (int m = 0; m < nb; ++m) {
            const uint32_t stage = cs;
            // the give-up is warp-uniform: no lane leaves while its warp-mates
            // go on to a __syncwarp
            if (!__all_sync(~0u, mbar_wait(full0 + 8u * stage, cph, A.wait_ns))) {
                if (lane == 0) record(A.status, 1);
                return;
            }
            if (++cs == (uint32_t)S) {
                cs = 0;
                cph ^= 1u;
            }
            RawVecs<K, CB16, U> raw;
            if (full_tile && mine) {
#pragma unroll
                for (int v = 0; v < U; ++v)
#pragma unroll
                    for (int j = 0; j < K; ++j) {
                        const unsigned char* p = chunk(stage, j) + (size_t)(ev[v] - e0) * ES;
                        raw[v][j][0] = *reinterpret_cast<const uint4*>(p);
                        if constexpr (!CB16) raw[v][j][CB16 ? 0 : 1] = *reinterpret_cast<const uint4*>(p + 16);
                    }
            }
            // gates of this member (staged rows or global memory), read as
            // each vector is accumulated
            const void* gp = GATED ? A.m_gate[first + m] : nullptr;
            if (GATED && gp && A.stage_gate_bytes) gp = gate_stage(stage);
            auto gate = [&](int v, float (&gv)[8]) {
                if (gp)
                    load_x8(gp, A.gate_bf16, (long long)gi[v], gv);
                else
#pragma unroll
                    for (int e = 0; e < 8; ++e) gv[e] = 1.0f;
            };
            // prediction-only launches release the stage as soon as it is read
            // and recompute guarded elements from registers; grouped launches
            // and bf16 ones with K >= 7 keep the stage until the member is done
            // and recompute from shared memory, which frees the history values'
            // registers early (bf16 K >= 7 would otherwise spill under the cap)
            if (!LATE) release_stage(empty0 + 8u * stage, lane);
            if (full_tile && mine) {
                void* out = member_out<K, CB16, U>(A, first + m, ev, raw);
                if constexpr (ONE) {
                    if (resid != nullptr) member_one<K, CB16, U, GATED>(raw, acc, gate);
                } else if (A.precise) {
                    member_precise<K, CB16, U, GATED>(A, out, ev, raw, resid != nullptr, acc, gate);
                } else if constexpr (LATE) {
                    auto exact = [&](int v, int e, float& hi, float& lo) {
                        const size_t off = (size_t)(ev[v] - e0 + e) * ES;
                        float p = 0.0f, cc = 0.0f;
#pragma unroll
                        for (int j = 0; j < K; ++j) {
                            const unsigned char* src = chunk(stage, j) + off;
                            const float f = CB16 ? __uint_as_float((uint32_t)(*reinterpret_cast<const uint16_t*>(src)) << 16)
                                                 : *reinterpret_cast<const float*>(src);
                            dot2_step(A.w_hi[j], A.w_lo[j], f, p, cc);
                        }
                        two_sum(p, cc, hi, lo);
                    };
                    member_fast<K, CB16, U, false, GATED>(A, A.m_off[first + m], out, ev, raw, resid != nullptr,
                                                          acc, gate, exact);
                } else {
                    member_fast<K, CB16, U, true, GATED>(A, A.m_off[first + m], out, ev, raw, resid != nullptr,
                                                         acc, gate);
                }
            }
            if (LATE && !hold) release_stage(empty0 + 8u * stage, lane);
        }
        if (GROUPED && hold) {
            const uint32_t last = stage_of(nb - 1);
            auto xload = [&](int v, float (&x)[8]) {
                if (A.stage_x)
                    unpack_bf16x8(*reinterpret_cast<const uint4*>(chunk(last, K) + (size_t)(ev[v] - e0) * 2), x);
                else
                    load_x8(resid, A.resid_bf16, ev[v], x);
            };
            if (!mine) {
            } else if (!ONE && A.precise) {
                resid_precise<U>(A, ev, acc, resid, xload);
            } else {
                // Dot2 of x + sum_b P_b for one element, from the held stages
                auto exact = [&](int v, int e, float xe, float& hi, float& lo) {
                    const size_t off = (size_t)(ev[v] - e0 + e) * ES;
                    float tp = xe, tc = 0.0f;
                    for (int m = 0; m < nb; ++m) {
                        const uint32_t st = stage_of(m);
                        float p = 0.0f, cc = 0.0f, h, l, qq;
#pragma unroll
                        for (int j = 0; j < K; ++j) {
                            const unsigned char* src = chunk(st, j) + off;
                            const float f = CB16 ? __uint_as_float((uint32_t)(*reinterpret_cast<const uint16_t*>(src)) << 16)
                                                 : *reinterpret_cast<const float*>(src);
                            dot2_step(A.w_hi[j], A.w_lo[j], f, p, cc);
                        }
                        two_sum(p, cc, h, l);
                        // a member without a gate adds like an ungated one (as exact_resid)
                        const void* gm = GATED ? A.m_gate[first + m] : nullptr;
                        if (gm) {
                            const float gv = load_elem(A.stage_gate_bytes ? gate_stage(st) : gm, A.gate_bf16, gi[v] + e);
                            add_gated_pair(gv, h, l, tp, tc);
                        } else {
                            two_sum(tp, h, tp, qq);
                            tc = __fadd_rn(tc, __fadd_rn(qq, l));
                        }
                    }
                    two_sum(tp, tc, hi, lo);
                };
                resid_fast<K, U>(A, it, ev, acc, resid, xload, exact, ONE ? A.w_guard[0] : 1.0f);
            }
            fence_generic_to_async();
            __syncwarp();
            if (lane == 0)
                for (int m = 0; m < nb; ++m) mbar_arrive(empty0 + 8u * stage_of(m));
        } else if (!full_tile) {
            const long long end = e0 + TE < numel ? e0 + TE : numel;
            for (long long e = e0 + c; e < end; e += NCT) scalar_element<CB16>(A, K, it, e);
        }
    }
}

}  // namespace
}  // namespace cbk
