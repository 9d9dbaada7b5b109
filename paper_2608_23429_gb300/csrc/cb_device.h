// Internal: kernel argument blocks and launchers shared by the host plan
// (plan.cpp) and the kernels (extrapolate*.cu, epilogue.cu, push.cu), and the
// library's own status block (static_status.cu). Not part of the ABI.
#pragma once

#include <cuda_runtime.h>

#include <cstdint>

namespace cbk {

constexpr int kThreads = 256;     // threads per CTA
constexpr int kVecElems = 8;      // elements per vector (16 B of bf16, 32 B of fp32)
constexpr int kMaxItems = 256;    // work items (tensors, or residual groups) per launch
constexpr int kMaxMembers = 256;  // branch tensors per launch

// Vectors each thread handles per tile: two 16-B vectors for a bf16 cache,
// one 32-B vector for an fp32 cache (both give 2*K 16-B loads in flight).
__host__ __device__ constexpr int vectors_per_thread(bool cache_bf16) { return cache_bf16 ? 2 : 1; }
__host__ __device__ constexpr long long tile_elems(bool cache_bf16) {
    return (long long)kThreads * vectors_per_thread(cache_bf16) * kVecElems;
}

// One skipped-step launch. Items are the units of work: a single branch
// tensor, or (with hidden states) all branch tensors of one residual group.
// Every item is cut into tiles of tile_elems() elements; tiles are numbered
// consecutively across items and dealt to a persistent grid.
struct ExtrapArgs {
    // byte address of the history: entry j of member m starts at
    // hist_base + slot_off[j] + m_off[m] (the ring arena and offsets inside it;
    // for a full step's epilogue, base 0 and m_off the new features' addresses)
    unsigned long long hist_base;
    long long slot_off[8];       // byte offset of history entry j (0 = oldest)
    float w_hi[8];               // fp32(w_j)
    float w_lo[8];               // fp32(w_j - w_hi[j])
    float w_guard[8];            // (K+2) u (1.01) 2^9 |w_hi[j]|: the fast path's scaled error bound
    int n_items;
    int tiles_total;
    int out_bf16;    // predictions are bf16 (else fp32)
    int resid_bf16;  // hidden states are bf16 (else fp32)
    int precise;     // 1: compensated (Dot2) arithmetic for every element
    int copy_out;    // full-step epilogue: outputs receive the (K = 1) sources converted, not a prediction
    int stages;                  // bulk variant: shared-memory pipeline depth
    int stage_chunks;            // bulk variant: 8 KB chunks per stage (K, or K + 1 with hidden states)
    int stage_x;                 // bulk variant: bf16 hidden states are staged as chunk K
    unsigned stage_gate_bytes;   // bulk variant: bytes per stage for gate rows (0: gates read from global)
    unsigned long long wait_ns;  // bulk variant: limit of every barrier wait
    int* status;                 // bulk variant: device status word (codes OR-ed in)
    int withhold_first;          // bulk variant, tests only: announce but never issue the first copies
    int tile_begin[kMaxItems + 1];
    long long numel[kMaxItems];
    void* resid[kMaxItems];           // hidden state of the item, or null
    unsigned char nb[kMaxItems];      // member tensors of the item
    unsigned char vec_ok[kMaxItems];  // every pointer of the item is 16-B aligned
    short first[kMaxItems];           // first member index
    long long m_off[kMaxMembers];     // byte offset of the member tensor inside one slot
    void* m_out[kMaxMembers];         // prediction output of the member, or null
    // gated hidden-state update (x <- x + sum_b g_b * P_b); read by gated kernels only
    int gate_bf16;                      // gates are bf16 (else fp32)
    const void* m_gate[kMaxMembers];    // gate [batch, hidden] of the member, or null (gate 1)
    unsigned i_hidden[kMaxItems];       // hidden size of the item's tensors
    unsigned i_row[kMaxItems];          // tokens * hidden of the item's tensors
    unsigned long long i_hidden_magic[kMaxItems];  // ceil(2^64 / i_hidden) (0: i_hidden = 1)
    unsigned long long i_row_magic[kMaxItems];     // ceil(2^64 / i_row) (0: i_row = 1)
};

// One full-step launch: copy/convert every tensor into one ring slot.
struct PushArgs {
    unsigned char* slot;  // base of the destination slot
    int n_items;
    int tiles_total;
    int tile_begin[kMaxItems + 1];
    long long numel[kMaxItems];
    long long off[kMaxItems];  // byte offset of the tensor inside the slot
    const void* src[kMaxItems];
    unsigned char vec_ok[kMaxItems];
};

constexpr long long push_tile_elems = (long long)kThreads * 2 * kVecElems;


cudaError_t launch_extrapolate(const ExtrapArgs& a, int K, bool cache_bf16, int grid, cudaStream_t s);
// gated variant of the direct kernel (extrapolate_gated.cu)
cudaError_t launch_extrapolate_gated(const ExtrapArgs& a, int K, bool cache_bf16, int grid, cudaStream_t s);
cudaError_t extrapolate_blocks_per_sm(int K, bool cache_bf16, int* blocks);

// Bulk-copy pipeline variant (extrapolate_bulk.cu). Its barrier block holds
// the full and empty barriers of at most kMaxStages stages.
constexpr int kMaxStages = 16;
// CTAs per SM of the bulk kernel (two of 8 consumer warps each, else one):
// two for K = 1, for bf16 prediction-only launches (not `grouped`) with
// K <= 2 and for ungated bf16 grouped launches with K = 2..3, where two
// vectors per thread still fit the register budget. Ungated bf16 grouped
// launches with K = 1 (the full-step epilogue from bf16 features) stream
// faster as one CTA of 16 warps (GB300: FLUX 88.3 -> 94.1 %, DiT-256
// 81.2 -> 90.1 % of the copy peak, PixArt unchanged); gated ones do not
// (DiT-256 88.0 -> 63.9 %) and keep two.
__host__ __device__ constexpr int bulk_ctas_per_sm(int K, bool src_bf16, bool grouped, bool gated) {
    return ((K == 1 && !(src_bf16 && grouped && !gated)) || (src_bf16 && !grouped && K <= 2) ||
            (src_bf16 && grouped && !gated && K >= 2 && K <= 3))
               ? 2
               : 1;
}
size_t bulk_smem_bytes(int chunks_per_stage, size_t extra_per_stage, int stages);
cudaError_t prepare_extrapolate_bulk(int K, bool cache_bf16, size_t smem);
// grouped: some item updates a hidden state or has several members (the
// kernel's hidden-state bookkeeping); it also selects the CTA shape.
cudaError_t launch_extrapolate_bulk(const ExtrapArgs& a, int K, bool cache_bf16, bool grouped, int grid, size_t smem,
                                    cudaStream_t s);
// gated variant of the bulk kernel (extrapolate_bulk_gated.cu)
cudaError_t prepare_extrapolate_bulk_gated(int K, bool cache_bf16, size_t smem);
cudaError_t launch_extrapolate_bulk_gated(const ExtrapArgs& a, int K, bool cache_bf16, int grid, size_t smem,
                                          cudaStream_t s);

// Full-step epilogue kernel (epilogue.cu) for ungated bf16 features: a
// one-entry history of weight 1 on 2048-element tiles, one 8-element vector
// per thread and tile.
constexpr long long epilogue_tile_elems = (long long)kThreads * kVecElems;
cudaError_t launch_epilogue(const ExtrapArgs& a, int grid, cudaStream_t s);
cudaError_t epilogue_blocks_per_sm(int* blocks);

cudaError_t launch_push(const PushArgs& a, bool src_bf16, bool dst_bf16, int grid, cudaStream_t s);
cudaError_t push_blocks_per_sm(bool src_bf16, bool dst_bf16, int* blocks);

// Status word of cb_extrapolate_noalloc in the library's own device block
// (static_status.cu): its device address on `device`, which must be the
// current device. The first call per device looks the address up.
constexpr int kMaxStatusDevices = 64;
cudaError_t noalloc_status_word(int device, int** word);

}  // namespace cbk
