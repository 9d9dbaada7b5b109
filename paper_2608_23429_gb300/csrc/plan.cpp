// Host side of libchebboost: the plan (the offline weight precomputation of
// Sec. 3.3; Alg. 1 offline stage), the history buffer's ring bookkeeping, the
// online weights (Sec. 3.2 Eq. barycentric_coeff) and the kernel launches.
// Everything here is fp64 host arithmetic that runs in microseconds per call;
// all device work is in push.cu (cache write), epilogue.cu (full-step
// epilogue) and the extrapolate*.cu instantiations of the skipped-step kernels.
#include <cuda_runtime.h>

#include <algorithm>
#include <cmath>
#include <cstdint>
#include <cstring>
#include <memory>
#include <new>
#include <string>
#include <vector>

#include "../../include/chebboost.h"
#include "cb_device.h"

namespace {

thread_local std::string g_last_error;

int cuda_fail(cudaError_t e, const char* where) {
    g_last_error = std::string(where) + ": " + cudaGetErrorName(e) + ": " + cudaGetErrorString(e);
    return CB_ERR_CUDA;
}

size_t esize(cb_dtype d) { return d == CB_BF16 ? 2 : 4; }
bool valid_dtype(cb_dtype d) { return d == CB_BF16 || d == CB_FP32; }
size_t round_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

// Barycentric weights rho_j = 1 / prod_{k != j} (x_j - x_k) (App. A, Eq. general_weights).
bool rho_of(const double* x, int n, double* rho) {
    for (int j = 0; j < n; ++j) {
        double d = 1.0;
        for (int k = 0; k < n; ++k)
            if (k != j) d *= x[j] - x[k];
        if (d == 0.0 || !std::isfinite(d)) return false;
        rho[j] = 1.0 / d;
    }
    return true;
}

// Interpolation coefficients w_j = (rho_j / (x - x_j)) / sum_i rho_i / (x - x_i)
// (Sec. 3.2, Eq. barycentric_coeff). A target on a node gives the unit vector.
void coeff_of(const double* x, const double* rho, int n, double xq, double* w) {
    for (int j = 0; j < n; ++j)
        if (xq == x[j]) {
            for (int i = 0; i < n; ++i) w[i] = (i == j) ? 1.0 : 0.0;
            return;
        }
    double den = 0.0;
    for (int i = 0; i < n; ++i) {
        w[i] = rho[i] / (xq - x[i]);
        den += w[i];
    }
    for (int i = 0; i < n; ++i) w[i] /= den;
}

struct DeviceInfo {
    int device = -1;
    int sms = 0;
    int smem_optin = 0;                    // largest dynamic shared memory per CTA
    int smem_per_sm = 0;                   // shared memory of one SM
    int occ_extrap[2][CB_MAX_K + 1] = {};  // [cache_bf16][K]
    int occ_push[2][2] = {};               // [src_bf16][dst_bf16]
    int occ_epilogue = 0;                  // epilogue kernel (bf16 features, no gates)
    int bulk_stages[2][CB_MAX_K + 1] = {};  // 1 once the kernel's shared-memory limit is raised
    int bulk_gated[2][CB_MAX_K + 1] = {};   // the same for the gated kernel
};

}  // namespace

struct cb_plan {
    int K = 0;
    cb_dtype cache_dtype = CB_BF16;
    double t_min = 0, t_max = 1;
    std::vector<cb_tensor_desc> tensors;
    std::vector<std::vector<int>> groups;  // residual group -> member tensors
    std::vector<double> node_t;            // full-step timesteps, sampling order
    std::vector<double> node_tau;
    int dir = 0;                           // +1 increasing, -1 decreasing t
    std::vector<double> rho_win;           // rho of node window i: rho_win[i*K + j]
    std::vector<long long> off;            // byte offset of tensor i inside a slot
    std::vector<long long> sh_tokens;      // [batch, tokens, hidden] of each tensor (0: unset)
    std::vector<long long> sh_hidden;
    size_t slot_bytes = 0;
    // bound history buffer
    unsigned char* cache = nullptr;
    // ring state of H
    double slot_t[CB_MAX_K] = {};
    int next = 0;   // slot written by the next push
    int count = 0;  // entries held (<= K)
    bool has_last = false;
    double last_t = 0;
    bool status_clear = false;  // the device status word was zeroed since binding
    int kernel = CB_KERNEL_AUTO;
    unsigned long long wait_ns = 1000000000ull;
    int withhold_first = 0;
    bool partial = false;  // extrapolate from fewer than K entries while H fills
    DeviceInfo dev;
    // value-initialised: no field of a launch's arguments is ever left unset
    std::unique_ptr<cbk::ExtrapArgs> eargs{new cbk::ExtrapArgs()};
    std::unique_ptr<cbk::PushArgs> pargs{new cbk::PushArgs()};

    double tau(double t) const { return 2.0 * (t - t_min) / (t_max - t_min) - 1.0; }
    int* status_word() const { return reinterpret_cast<int*>(cache + slot_bytes * (size_t)K); }
    int oldest() const { return count < K ? 0 : next; }
};

namespace {

int ensure_device(cb_plan* p) {
    int d = 0;
    cudaError_t e = cudaGetDevice(&d);
    if (e != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
    if (p->dev.device != d) {
        DeviceInfo info;
        info.device = d;
        e = cudaDeviceGetAttribute(&info.sms, cudaDevAttrMultiProcessorCount, d);
        if (e != cudaSuccess) return cuda_fail(e, "cudaDeviceGetAttribute");
        e = cudaDeviceGetAttribute(&info.smem_optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, d);
        if (e != cudaSuccess) return cuda_fail(e, "cudaDeviceGetAttribute");
        e = cudaDeviceGetAttribute(&info.smem_per_sm, cudaDevAttrMaxSharedMemoryPerMultiprocessor, d);
        if (e != cudaSuccess) return cuda_fail(e, "cudaDeviceGetAttribute");
        p->dev = info;
    }
    return CB_OK;
}

int extrap_grid(cb_plan* p, int K, bool cb16, int tiles, int* grid) {
    int& occ = p->dev.occ_extrap[cb16 ? 1 : 0][K];
    if (occ == 0) {
        cudaError_t e = cbk::extrapolate_blocks_per_sm(K, cb16, &occ);
        if (e != cudaSuccess || occ <= 0) {
            occ = 0;
            return cuda_fail(e == cudaSuccess ? cudaErrorInvalidConfiguration : e, "occupancy");
        }
    }
    long long g = (long long)p->dev.sms * occ;
    *grid = (int)(tiles < g ? tiles : g);
    return CB_OK;
}

// Largest gate staging per pipeline stage (two rows of 4096 fp32 channels).
constexpr size_t kMaxStagedGateBytes = 32768;

// Pipeline of the bulk kernel: as many stages of `chunks` 8 KB chunks (plus
// `extra` bytes) as fit in one CTA's shared memory, at most kMaxStages, and
// the CTAs per SM. A shape made for two CTAs per SM runs one, with all of the
// SM's shared memory, when half of it cannot hold `min_stages`. The kernel's
// dynamic shared-memory limit is raised to the device maximum once per
// instantiation.
int bulk_config(cb_plan* p, int K, bool cb16, bool grouped, int chunks, size_t extra, bool gated, int min_stages,
                int* stages, size_t* smem, int* ctas_per_sm) {
    int& prepared = gated ? p->dev.bulk_gated[cb16 ? 1 : 0][K] : p->dev.bulk_stages[cb16 ? 1 : 0][K];
    if (prepared == 0) {
        cudaError_t e = gated ? cbk::prepare_extrapolate_bulk_gated(K, cb16, (size_t)p->dev.smem_optin)
                              : cbk::prepare_extrapolate_bulk(K, cb16, (size_t)p->dev.smem_optin);
        if (e != cudaSuccess) return cuda_fail(e, "cudaFuncSetAttribute");
        prepared = 1;
    }
    // with several CTAs per SM each gets its share of the SM's shared memory
    // (less the 1 KB the hardware reserves per CTA)
    for (int per_sm = cbk::bulk_ctas_per_sm(K, cb16, grouped, gated); per_sm >= 1; --per_sm) {
        size_t cap = (size_t)p->dev.smem_optin;
        if (per_sm > 1) cap = std::min(cap, (size_t)p->dev.smem_per_sm / per_sm - 1024);
        int s = cbk::kMaxStages;
        while (s > 1 && cbk::bulk_smem_bytes(chunks, extra, s) > cap) --s;
        *stages = cbk::bulk_smem_bytes(chunks, extra, s) <= cap ? s : 0;
        *smem = cbk::bulk_smem_bytes(chunks, extra, s);
        *ctas_per_sm = per_sm;
        if (*stages >= min_stages) break;
    }
    return CB_OK;
}

int push_grid(cb_plan* p, bool sb, bool db, int tiles, int* grid) {
    int& occ = p->dev.occ_push[sb ? 1 : 0][db ? 1 : 0];
    if (occ == 0) {
        cudaError_t e = cbk::push_blocks_per_sm(sb, db, &occ);
        if (e != cudaSuccess || occ <= 0) {
            occ = 0;
            return cuda_fail(e == cudaSuccess ? cudaErrorInvalidConfiguration : e, "occupancy");
        }
    }
    // fewer concurrent copy streams stream faster than full occupancy (FLUX
    // cache writes: bf16 sources best at 4 CTAs per SM, fp32 sources at 3)
    const int cap = sb ? 4 : 3;
    long long g = (long long)p->dev.sms * (occ < cap ? occ : cap);
    *grid = (int)(tiles < g ? tiles : g);
    return CB_OK;
}

bool aligned(const void* ptr, size_t a) { return ((uintptr_t)ptr % a) == 0; }

// Multiplier of the kernels' division by d < 2^32: ceil(2^64 / d), 0 for d <= 1.
unsigned long long div_magic(unsigned d) { return d <= 1 ? 0ull : ~0ull / d + 1ull; }

// Logical history window: n entries, oldest first, with the slot of each.
struct Window {
    int n;
    double t[CB_MAX_K];
    double tau[CB_MAX_K];
    int slot[CB_MAX_K];
};

// rho for a window: reuse the offline table when the window is K consecutive
// nodes of the plan, otherwise compute it the same way now.
bool window_rho(const cb_plan* p, const Window& w, double* rho) {
    const int K = p->K;
    const int n = (int)p->node_t.size();
    if (w.n == K) {
        for (int i = 0; i + K <= n; ++i) {
            if (p->node_t[i] != w.t[0]) continue;
            bool match = true;
            for (int j = 1; j < K && match; ++j) match = p->node_t[i + j] == w.t[j];
            if (match) {
                std::memcpy(rho, &p->rho_win[(size_t)i * K], sizeof(double) * K);
                return true;
            }
        }
    }
    return rho_of(w.tau, w.n, rho);
}

int weights_for(const cb_plan* p, const Window& w, double t_target, double* out) {
    if (!std::isfinite(t_target)) return CB_ERR_ARG;
    double rho[CB_MAX_K];
    if (!window_rho(p, w, rho)) return CB_ERR_NODES_DEGENERATE;
    for (int j = 0; j < w.n; ++j)
        if (t_target == w.t[j]) {  // the target is a cached node: return it exactly
            for (int i = 0; i < w.n; ++i) out[i] = (i == j) ? 1.0 : 0.0;
            return CB_OK;
        }
    coeff_of(w.tau, rho, w.n, p->tau(t_target), out);
    return CB_OK;
}

// Entries a skipped step may use: all K once H is full; with partial history
// enabled, whatever H holds (at least one); otherwise none.
int live_entries(const cb_plan* p) {
    if (p->count == p->K) return p->K;
    if (p->partial && p->count >= 1) return p->count;
    return 0;
}

Window live_window(const cb_plan* p, int n) {
    Window w{};
    w.n = n;
    const int o = p->oldest();
    for (int j = 0; j < n; ++j) {
        w.slot[j] = (o + j) % p->K;
        w.t[j] = p->slot_t[w.slot[j]];
        w.tau[j] = p->tau(w.t[j]);
    }
    return w;
}

// Gates (one per tensor, [batch, hidden] of gate_dtype, null = 1) apply to the
// hidden-state update of a grouped tensor: its shape must be set, its group's
// tensors must share it, and indexing stays in 32 bits.
int check_gates(const cb_plan* p, const void* const* gates, cb_dtype gate_dtype) {
    if (!gates) return CB_OK;
    if (!valid_dtype(gate_dtype)) return CB_ERR_ARG;
    const int n = (int)p->tensors.size();
    for (int i = 0; i < n; ++i) {
        if (!gates[i]) continue;
        if (p->sh_hidden[i] <= 0) return CB_ERR_ARG;  // cb_plan_set_shapes first
        if (!aligned(gates[i], esize(gate_dtype))) return CB_ERR_ALIGN;
        if (p->tensors[i].numel > 0xFFFFFFFFLL) return CB_ERR_LIMIT;
    }
    return CB_OK;
}

// The device status word is zeroed once after binding, on the stream of the
// first launch, after that launch's arguments have all been validated.
int clear_status_once(cb_plan* p, void* stream) {
    if (p->status_clear) return CB_OK;
    cudaError_t e = cudaMemsetAsync(p->status_word(), 0, sizeof(int), (cudaStream_t)stream);
    if (e != cudaSuccess) return cuda_fail(e, "cudaMemsetAsync");
    p->status_clear = true;
    return CB_OK;
}

// A history buffer given with the call instead of the bound arena, and the
// status word its launch records into (cb_extrapolate_noalloc). `launched` is
// set once the word has been cleared for a launch.
struct CallerHistory {
    const unsigned char* hist;
    int* status;
    bool launched;
};

// Zero a status word that every call shares, on the launch's stream.
int clear_word(int* word, void* stream) {
    cudaError_t e = cudaMemsetAsync(word, 0, sizeof(int), (cudaStream_t)stream);
    return e == cudaSuccess ? CB_OK : cuda_fail(e, "cudaMemsetAsync");
}

// One skipped-step launch over the window `win` with the fp64 weights w[0..n).
// With `feats` it is instead a full step's epilogue: a one-entry history (the
// new features, weight 1) whose members are written, converted, into the ring
// slot `next` while the hidden states receive x + sum_b g_b f_b. With `ch` the
// window's slots are read from ch->hist and events recorded in ch->status.
int run_launch(cb_plan* p, const Window& win, const double* w, void* const* outs, cb_dtype out_dtype,
               void* const* resid, cb_dtype resid_dtype, void* stream, const void* const* gates = nullptr,
               cb_dtype gate_dtype = CB_BF16, const void* const* feats = nullptr, cb_dtype feat_dtype = CB_BF16,
               CallerHistory* ch = nullptr) {
    if (!ch && !p->cache) return CB_ERR_UNBOUND;
    const int K = win.n;
    if (K < 1 || (!feats && !ch && p->count < K)) return CB_ERR_HISTORY_NOT_FULL;
    if (!valid_dtype(out_dtype) || !valid_dtype(resid_dtype)) return CB_ERR_ARG;
    const int n = (int)p->tensors.size();
    const int ng = (int)p->groups.size();
    const size_t oes = esize(out_dtype), res = esize(resid_dtype);
    if (outs)
        for (int i = 0; i < n; ++i)
            if (outs[i] && !aligned(outs[i], oes)) return CB_ERR_ALIGN;
    if (resid)
        for (int g = 0; g < ng; ++g)
            if (resid[g] && !aligned(resid[g], res)) return CB_ERR_ALIGN;

    for (int j = 0; j < K; ++j)
        if (!std::isfinite(w[j])) return CB_ERR_ARG;
    int rc = check_gates(p, gates, gate_dtype);
    if (rc != CB_OK) return rc;

    cbk::ExtrapArgs& A = *p->eargs;
    // the kernels' source type: the cache's, or the new features'
    const bool cb16 = (feats ? feat_dtype : p->cache_dtype) == CB_BF16;
    // A full step's epilogue runs its own kernel (unless CB_OPT_KERNEL names
    // one) when its threads keep enough loads in flight: ungated bf16 features
    // with every tensor in a residual group of three or more branches.
    // Otherwise the bulk pipeline streams faster (see epilogue.cu).
    bool epilogue = feats && p->kernel == CB_KERNEL_AUTO && feat_dtype == CB_BF16 && resid;
    for (int i = 0; epilogue && i < n; ++i) {
        const int g = p->tensors[i].group;
        epilogue = g >= 0 && resid[g] && p->groups[g].size() >= 3 && !(gates && gates[i]);
    }
    const long long te_bulk = cbk::tile_elems(cb16);
    const long long te = epilogue ? cbk::epilogue_tile_elems : te_bulk;
    unsigned char* slot = p->cache + (size_t)p->next * p->slot_bytes;
    A.hist_base = feats ? 0ull : (unsigned long long)(uintptr_t)(ch ? ch->hist : p->cache);
    A.copy_out = feats ? 1 : 0;
    for (int j = 0; j < CB_MAX_K; ++j) {
        const bool on = j < K;
        A.slot_off[j] = on && !feats ? (long long)win.slot[j] * (long long)p->slot_bytes : 0;
        const float hi = on ? (float)w[j] : 0.0f;
        A.w_hi[j] = hi;
        A.w_lo[j] = on ? (float)(w[j] - (double)hi) : 0.0f;
        // the fast path's bound, scaled: (K+2) u (1.01) 2^9 |w_hi[j]|, u = 2^-24
        A.w_guard[j] = (float)(std::fabs((double)hi) * (K + 2) * 1.01 * std::ldexp(1.0, -15));
    }
    A.out_bf16 = out_dtype == CB_BF16;
    A.resid_bf16 = resid_dtype == CB_BF16;

    int items = 0, members = 0;
    long long tiles = 0;
    bool any_out = false, any_resid = false;
    bool any_gate = false;
    A.gate_bf16 = gate_dtype == CB_BF16;
    auto add_item = [&](const int* mem, int nm, void* res_ptr) {
        const long long numel = p->tensors[mem[0]].numel;
        bool vec = !res_ptr || aligned(res_ptr, 16);
        A.first[items] = (short)members;
        A.i_hidden[items] = (unsigned)p->sh_hidden[mem[0]];
        A.i_row[items] = (unsigned)(p->sh_tokens[mem[0]] * p->sh_hidden[mem[0]]);
        A.i_hidden_magic[items] = div_magic(A.i_hidden[items]);
        A.i_row_magic[items] = div_magic(A.i_row[items]);
        for (int m = 0; m < nm; ++m) {
            const int i = mem[m];
            void* o = feats ? slot + p->off[i] : outs ? outs[i] : nullptr;
            const void* g = (res_ptr && gates) ? gates[i] : nullptr;
            A.m_off[members] = feats ? (long long)(uintptr_t)feats[i] : p->off[i];
            if (feats) vec = vec && aligned(feats[i], 16);
            A.m_out[members] = o;
            A.m_gate[members] = g;
            if (g) {  // vectors of 8 stay inside one gate row
                any_gate = true;
                vec = vec && aligned(g, 16) && p->sh_hidden[i] % 8 == 0;
            }
            if (o) {
                any_out = true;
                vec = vec && aligned(o, 16);
            }
            ++members;
        }
        if (res_ptr) any_resid = true;
        A.nb[items] = (unsigned char)nm;
        A.resid[items] = res_ptr;
        A.vec_ok[items] = vec ? 1 : 0;
        A.numel[items] = numel;
        A.tile_begin[items] = (int)tiles;
        tiles += (numel + te - 1) / te;
        ++items;
    };
    std::vector<char> in_group(n, 0);
    if (resid)
        for (int g = 0; g < ng; ++g)
            if (resid[g] && !p->groups[g].empty()) {
                add_item(p->groups[g].data(), (int)p->groups[g].size(), resid[g]);
                for (int i : p->groups[g]) in_group[i] = 1;
            }
    for (int i = 0; i < n; ++i)
        if (!in_group[i] && (feats || (outs && outs[i]))) add_item(&i, 1, nullptr);
    if (tiles > 0x7FFFFFFFLL) return CB_ERR_LIMIT;
    A.tile_begin[items] = (int)tiles;
    A.n_items = items;
    A.tiles_total = (int)tiles;
    // a full step's slot write is a conversion, not arithmetic
    A.precise = (any_out && !feats && out_dtype == CB_FP32) || (any_resid && resid_dtype == CB_FP32);
    if (items == 0) return CB_OK;  // nothing requested

    A.wait_ns = p->wait_ns;
    A.status = ch ? ch->status : p->status_word();
    A.withhold_first = p->withhold_first;
    A.stages = 0;
    A.stage_chunks = K;
    A.stage_x = 0;
    A.stage_gate_bytes = 0;

    rc = ensure_device(p);
    if (rc != CB_OK) return rc;
    auto clear_status = [&]() {
        if (!ch) return clear_status_once(p, stream);
        const int r = clear_word(ch->status, stream);
        ch->launched = r == CB_OK;
        return r;
    };
    auto launch_direct = [&]() {
        int grid = 0;
        int r = extrap_grid(p, K, cb16, (int)tiles, &grid);
        if (r != CB_OK) return r;
        r = clear_status();
        if (r != CB_OK) return r;
        cudaError_t e = any_gate ? cbk::launch_extrapolate_gated(A, K, cb16, grid, (cudaStream_t)stream)
                                 : cbk::launch_extrapolate(A, K, cb16, grid, (cudaStream_t)stream);
        if (e != cudaSuccess) return cuda_fail(e, "extrapolate launch");
        return (int)CB_OK;
    };
    if (epilogue) {
        int& occ = p->dev.occ_epilogue;
        if (occ == 0) {
            cudaError_t e = cbk::epilogue_blocks_per_sm(&occ);
            if (e != cudaSuccess || occ <= 0) {
                occ = 0;
                return cuda_fail(e == cudaSuccess ? cudaErrorInvalidConfiguration : e, "occupancy");
            }
        }
        const long long ctas = (long long)p->dev.sms * occ;
        const int grid = (int)(tiles < ctas ? tiles : ctas);
        rc = clear_status();
        if (rc != CB_OK) return rc;
        cudaError_t e = cbk::launch_epilogue(A, grid, (cudaStream_t)stream);
        if (e != cudaSuccess) return cuda_fail(e, "epilogue launch");
        return CB_OK;
    }
    if (p->kernel == CB_KERNEL_DIRECT) return launch_direct();
    // bf16 hidden states travel through shared memory with the last member of
    // their group; the pipeline must hold a whole group plus one stage ahead
    int max_nb = 1;
    for (int i = 0; i < items; ++i)
        if (A.nb[i] > max_nb) max_nb = A.nb[i];
    A.stage_x = any_resid && A.resid_bf16 ? 1 : 0;
    A.stage_chunks = K + A.stage_x;
    // gate rows travel with their member when every gated tile touches at
    // most two batches (a batch holds a tile or more) and two rows are small
    A.stage_gate_bytes = 0;
    if (any_gate) {
        const size_t gs = esize(gate_dtype);
        size_t need = 0;
        bool fits = true;
        for (int i = 0; i < items; ++i) {
            bool gated_item = false;
            for (int m = 0; m < A.nb[i]; ++m) gated_item = gated_item || A.m_gate[A.first[i] + m];
            if (!gated_item || !A.vec_ok[i]) continue;
            fits = fits && (long long)A.i_row[i] >= te_bulk;
            need = std::max(need, 2 * (size_t)A.i_hidden[i] * gs);
        }
        if (fits && need <= kMaxStagedGateBytes) A.stage_gate_bytes = (unsigned)((need + 127) / 128 * 128);
    }
    // the grouped kernel (hidden-state bookkeeping) for gates, hidden states or multi-member items
    bool grouped = any_gate;
    for (int i = 0; i < items; ++i) grouped = grouped || A.resid[i] != nullptr || A.nb[i] > 1;
    size_t smem = 0;
    int per_sm = 1;
    rc = bulk_config(p, K, cb16, grouped, A.stage_chunks, A.stage_gate_bytes, any_gate, max_nb + 1, &A.stages,
                     &smem, &per_sm);
    if (rc != CB_OK) return rc;
    if (A.stages < max_nb + 1) return launch_direct();  // too deep for shared memory
    // Persistent grid. bf16 prediction-only launches with K >= 3 stream faster
    // over 3/4 of the SMs (one CTA each) than over all of them (measured on
    // GB300, repeatable within 0.5 %: FLUX 99 -> 103 %, PixArt 96 -> 104 %,
    // DiT-512 95 -> 101 % of the copy peak). Launches that update hidden states
    // are bound by their consumers and use every SM.
    double frac = 1.0;
    if (cb16 && !grouped && K >= 3) frac = 0.75;
    const long long ctas = std::max(1LL, (long long)((double)p->dev.sms * per_sm * frac));
    const int grid = (int)(tiles < ctas ? tiles : ctas);
    rc = clear_status();
    if (rc != CB_OK) return rc;
    cudaError_t e = any_gate ? cbk::launch_extrapolate_bulk_gated(A, K, cb16, grid, smem, (cudaStream_t)stream)
                             : cbk::launch_extrapolate_bulk(A, K, cb16, grouped, grid, smem, (cudaStream_t)stream);
    if (e != cudaSuccess) return cuda_fail(e, "extrapolate launch");
    return CB_OK;
}

}  // namespace

extern "C" {

int cb_schedule_full(int T, int r, int s0, int s1, int K, uint8_t* is_full, int* n_full) {
    if (T <= 0 || r <= 0 || s0 < 0 || s1 < 0 || K < 0 || !is_full) return CB_ERR_ARG;
    int held = 0, nf = 0;
    for (int s = 0; s < T; ++s) {
        const bool in_range = s >= s0 && s <= T - 1 - s1;
        bool full = !in_range || (s - s0) % r == 0;
        if (held < K) full = true;  // not enough history to extrapolate yet
        is_full[s] = full ? 1 : 0;
        if (full) {
            ++nf;
            if (held < K) ++held;
        }
    }
    if (n_full) *n_full = nf;
    return CB_OK;
}

int cb_plan_create(const double* node_t, int n_nodes, int K, const cb_tensor_desc* tensors, int n_tensors,
                   cb_dtype cache_dtype, double t_min, double t_max, cb_plan** out) {
    if (!out) return CB_ERR_ARG;
    *out = nullptr;
    if (K < 1 || K > CB_MAX_K) return K < 1 ? CB_ERR_ARG : CB_ERR_LIMIT;
    if (!node_t || n_nodes < K || !tensors || n_tensors < 1) return CB_ERR_ARG;
    if (n_tensors > CB_MAX_TENSORS) return CB_ERR_LIMIT;
    if (!valid_dtype(cache_dtype)) return CB_ERR_ARG;
    if (!(std::isfinite(t_min) && std::isfinite(t_max) && t_min < t_max)) return CB_ERR_ARG;
    for (int i = 0; i < n_nodes; ++i)
        if (!std::isfinite(node_t[i])) return CB_ERR_ARG;
    int dir = 0;
    if (n_nodes >= 2) {
        for (int i = 1; i < n_nodes; ++i) {
            const double d = node_t[i] - node_t[i - 1];
            if (d == 0.0) return CB_ERR_NODES_DEGENERATE;
            const int s = d > 0 ? 1 : -1;
            if (dir == 0) dir = s;
            if (s != dir) return CB_ERR_ARG;  // nodes must be strictly monotone
        }
    }
    try {
        std::unique_ptr<cb_plan> p(new cb_plan);
        p->K = K;
        p->cache_dtype = cache_dtype;
        p->t_min = t_min;
        p->t_max = t_max;
        p->dir = dir;
        p->tensors.assign(tensors, tensors + n_tensors);
        int ng = 0;
        for (const auto& d : p->tensors) {
            if (d.numel <= 0 || d.reserved != 0 || d.group < -1) return CB_ERR_ARG;
            if (d.numel > CB_MAX_NUMEL) return CB_ERR_LIMIT;
            if (d.group + 1 > ng) ng = d.group + 1;
        }
        static_assert(cbk::kMaxItems == CB_MAX_TENSORS, "one work item per tensor or group");
        if (ng > cbk::kMaxItems) return CB_ERR_LIMIT;
        p->groups.assign(ng, {});
        for (int i = 0; i < n_tensors; ++i) {
            const auto& d = p->tensors[i];
            if (d.group < 0) continue;
            auto& g = p->groups[d.group];
            if (!g.empty() && p->tensors[g[0]].numel != d.numel) return CB_ERR_ARG;
            g.push_back(i);
            if ((int)g.size() > CB_MAX_BRANCHES) return CB_ERR_LIMIT;
        }
        p->node_t.assign(node_t, node_t + n_nodes);
        p->node_tau.resize(n_nodes);
        for (int i = 0; i < n_nodes; ++i) p->node_tau[i] = p->tau(node_t[i]);
        // offline stage: rho for every window of K consecutive nodes
        p->rho_win.resize((size_t)(n_nodes - K + 1) * K);
        for (int i = 0; i + K <= n_nodes; ++i)
            if (!rho_of(&p->node_tau[i], K, &p->rho_win[(size_t)i * K])) return CB_ERR_NODES_DEGENERATE;
        // slot layout: tensors back to back, each at a CB_CACHE_ALIGN boundary
        size_t o = 0;
        p->off.resize(n_tensors);
        for (int i = 0; i < n_tensors; ++i) {
            p->off[i] = (long long)o;
            o = round_up(o + (size_t)p->tensors[i].numel * esize(cache_dtype), CB_CACHE_ALIGN);
        }
        p->slot_bytes = o;
        p->sh_tokens.assign(n_tensors, 0);
        p->sh_hidden.assign(n_tensors, 0);
        *out = p.release();
        return CB_OK;
    } catch (const std::bad_alloc&) {
        return CB_ERR_LIMIT;
    }
}

size_t cb_plan_cache_bytes(const cb_plan* p) {
    return p ? p->slot_bytes * (size_t)p->K + CB_STATUS_BYTES : 0;
}

int cb_plan_bind_cache(cb_plan* p, void* dev_ptr, size_t bytes) {
    if (!p || !dev_ptr || bytes < cb_plan_cache_bytes(p)) return CB_ERR_ARG;
    if (!aligned(dev_ptr, CB_CACHE_ALIGN)) return CB_ERR_ALIGN;
    p->cache = static_cast<unsigned char*>(dev_ptr);
    p->next = p->count = 0;
    p->has_last = false;
    p->status_clear = false;  // zeroed on the stream of the first launch
    return CB_OK;
}

int cb_cache_push(cb_plan* p, const void* const* feats, cb_dtype feat_dtype, double t, void* stream) {
    if (!p || !feats || !valid_dtype(feat_dtype) || !std::isfinite(t)) return CB_ERR_ARG;
    if (!p->cache) return CB_ERR_UNBOUND;
    const int n = (int)p->tensors.size();
    const size_t fes = esize(feat_dtype);
    for (int i = 0; i < n; ++i) {
        if (!feats[i]) return CB_ERR_ARG;
        if (!aligned(feats[i], fes)) return CB_ERR_ALIGN;
    }
    if (p->has_last) {
        const double d = t - p->last_t;
        if (d == 0.0 || (p->dir != 0 && (d > 0 ? 1 : -1) != p->dir)) return CB_ERR_ORDER;
    }
    for (int j = 0; j < p->count; ++j)
        if (p->slot_t[(p->oldest() + j) % p->K] == t) return CB_ERR_NODES_DEGENERATE;

    cbk::PushArgs& A = *p->pargs;
    const bool sb = feat_dtype == CB_BF16, db = p->cache_dtype == CB_BF16;
    A.slot = p->cache + (size_t)p->next * p->slot_bytes;
    long long tiles = 0;
    for (int i = 0; i < n; ++i) {
        A.tile_begin[i] = (int)tiles;
        A.numel[i] = p->tensors[i].numel;
        A.off[i] = p->off[i];
        A.src[i] = feats[i];
        A.vec_ok[i] = aligned(feats[i], 16) ? 1 : 0;
        tiles += (p->tensors[i].numel + cbk::push_tile_elems - 1) / cbk::push_tile_elems;
    }
    if (tiles > 0x7FFFFFFFLL) return CB_ERR_LIMIT;
    A.tile_begin[n] = (int)tiles;
    A.n_items = n;
    A.tiles_total = (int)tiles;
    int rc = ensure_device(p);
    if (rc != CB_OK) return rc;
    int grid = 0;
    rc = push_grid(p, sb, db, (int)tiles, &grid);
    if (rc != CB_OK) return rc;
    rc = clear_status_once(p, stream);
    if (rc != CB_OK) return rc;
    cudaError_t e = cbk::launch_push(A, sb, db, grid, (cudaStream_t)stream);
    if (e != cudaSuccess) return cuda_fail(e, "push launch");
    // the pair (t, f_t) is now in H; the oldest entry was overwritten when full
    p->slot_t[p->next] = t;
    p->next = (p->next + 1) % p->K;
    if (p->count < p->K) ++p->count;
    p->has_last = true;
    p->last_t = t;
    return CB_OK;
}

int cb_extrapolate(cb_plan* p, double t_target, void* const* outs, cb_dtype out_dtype, void* const* resid,
                   cb_dtype resid_dtype, void* stream) {
    if (!p) return CB_ERR_ARG;
    const int n = live_entries(p);
    if (n == 0) return p->cache ? CB_ERR_HISTORY_NOT_FULL : CB_ERR_UNBOUND;
    const Window win = live_window(p, n);
    double w[CB_MAX_K];
    const int rc = weights_for(p, win, t_target, w);
    if (rc != CB_OK) return rc;
    return run_launch(p, win, w, outs, out_dtype, resid, resid_dtype, stream);
}

int cb_extrapolate_ring(cb_plan* p, const double* slot_t, int head, double t_target, void* const* outs,
                        cb_dtype out_dtype, void* const* resid, cb_dtype resid_dtype, void* stream) {
    if (!p || !slot_t || head < 0 || head >= (p ? p->K : 1)) return CB_ERR_ARG;
    if (p->count < p->K) return p->cache ? CB_ERR_HISTORY_NOT_FULL : CB_ERR_UNBOUND;
    Window win{};
    win.n = p->K;
    for (int j = 0; j < p->K; ++j) {
        win.slot[j] = (head + j) % p->K;
        win.t[j] = slot_t[win.slot[j]];
        if (!std::isfinite(win.t[j])) return CB_ERR_ARG;
        win.tau[j] = p->tau(win.t[j]);
        for (int i = 0; i < j; ++i)
            if (win.t[i] == win.t[j]) return CB_ERR_NODES_DEGENERATE;
    }
    double w[CB_MAX_K];
    const int rc = weights_for(p, win, t_target, w);
    if (rc != CB_OK) return rc;
    return run_launch(p, win, w, outs, out_dtype, resid, resid_dtype, stream);
}

int cb_extrapolate_noalloc(cb_plan* p, const void* hist, size_t hist_bytes, const double* slot_t, int head,
                           double t_target, void* const* outs, cb_dtype out_dtype, void* const* resid,
                           cb_dtype resid_dtype, int* status, void* stream) {
    if (!p || !hist || !slot_t || head < 0 || head >= p->K) return CB_ERR_ARG;
    if (!aligned(hist, CB_CACHE_ALIGN)) return CB_ERR_ALIGN;
    if (hist_bytes < p->slot_bytes * (size_t)p->K) return CB_ERR_ARG;  // the K slots, no status block
    Window win{};
    win.n = p->K;
    for (int j = 0; j < p->K; ++j) {
        win.slot[j] = (head + j) % p->K;
        win.t[j] = slot_t[win.slot[j]];
        if (!std::isfinite(win.t[j])) return CB_ERR_ARG;
        win.tau[j] = p->tau(win.t[j]);
        for (int i = 0; i < j; ++i)
            if (win.t[i] == win.t[j]) return CB_ERR_NODES_DEGENERATE;
    }
    double w[CB_MAX_K];
    int rc = weights_for(p, win, t_target, w);
    if (rc != CB_OK) return rc;
    // the library's status word on the current device (looked up on the first call there)
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
    if (dev >= cbk::kMaxStatusDevices) return CB_ERR_LIMIT;
    int* word = nullptr;
    e = cbk::noalloc_status_word(dev, &word);
    if (e != cudaSuccess) return cuda_fail(e, "cudaGetSymbolAddress");
    CallerHistory ch{static_cast<const unsigned char*>(hist), word, false};
    rc = run_launch(p, win, w, outs, out_dtype, resid, resid_dtype, stream, nullptr, CB_BF16, nullptr, CB_BF16, &ch);
    if (rc != CB_OK) return rc;
    if (status) {
        if (!ch.launched) {  // nothing was requested, so nothing ran
            *status = 0;
            return CB_OK;
        }
        e = cudaMemcpyAsync(status, word, sizeof(int), cudaMemcpyDeviceToHost, (cudaStream_t)stream);
        if (e != cudaSuccess) return cuda_fail(e, "status read-back");
    }
    return CB_OK;
}

int cb_extrapolate_weights(cb_plan* p, const double* w_logical, void* const* outs, cb_dtype out_dtype,
                           void* const* resid, cb_dtype resid_dtype, void* stream) {
    if (!p || !w_logical) return CB_ERR_ARG;
    const int n = live_entries(p);
    if (n == 0) return p->cache ? CB_ERR_HISTORY_NOT_FULL : CB_ERR_UNBOUND;
    return run_launch(p, live_window(p, n), w_logical, outs, out_dtype, resid, resid_dtype, stream);
}

int cb_plan_set_shapes(cb_plan* p, const int64_t* bth) {
    if (!p || !bth) return CB_ERR_ARG;
    const int n = (int)p->tensors.size();
    for (int i = 0; i < n; ++i) {
        const int64_t b = bth[3 * i], t = bth[3 * i + 1], h = bth[3 * i + 2];
        const int64_t numel = p->tensors[i].numel;
        // b * t * h == numel, tested by division so that no product overflows
        if (b <= 0 || t <= 0 || h <= 0 || h > numel || t > numel / h) return CB_ERR_ARG;
        if (numel % (t * h) != 0 || numel / (t * h) != b) return CB_ERR_ARG;
        if (t * h > 0xFFFFFFFFLL) return CB_ERR_LIMIT;
    }
    for (const auto& g : p->groups)  // members of a group share one hidden state, hence one shape
        for (int i : g)
            if (bth[3 * i + 1] != bth[3 * g[0] + 1] || bth[3 * i + 2] != bth[3 * g[0] + 2]) return CB_ERR_ARG;
    for (int i = 0; i < n; ++i) {
        p->sh_tokens[i] = bth[3 * i + 1];
        p->sh_hidden[i] = bth[3 * i + 2];
    }
    return CB_OK;
}

int cb_extrapolate_gated(cb_plan* p, double t_target, void* const* outs, cb_dtype out_dtype, void* const* resid,
                         cb_dtype resid_dtype, const void* const* gates, cb_dtype gate_dtype, void* stream) {
    if (!p) return CB_ERR_ARG;
    const int n = live_entries(p);
    if (n == 0) return p->cache ? CB_ERR_HISTORY_NOT_FULL : CB_ERR_UNBOUND;
    const Window win = live_window(p, n);
    double w[CB_MAX_K];
    const int rc = weights_for(p, win, t_target, w);
    if (rc != CB_OK) return rc;
    return run_launch(p, win, w, outs, out_dtype, resid, resid_dtype, stream, gates, gate_dtype);
}

int cb_cache_push_residual(cb_plan* p, const void* const* feats, cb_dtype feat_dtype, double t, void* const* resid,
                           cb_dtype resid_dtype, const void* const* gates, cb_dtype gate_dtype, void* stream) {
    if (!p || !feats || !valid_dtype(feat_dtype) || !valid_dtype(resid_dtype) || !std::isfinite(t))
        return CB_ERR_ARG;
    if (!p->cache) return CB_ERR_UNBOUND;
    const int n = (int)p->tensors.size();
    const int ng = (int)p->groups.size();
    const size_t fes = esize(feat_dtype), res = esize(resid_dtype);
    for (int i = 0; i < n; ++i) {
        if (!feats[i]) return CB_ERR_ARG;
        if (!aligned(feats[i], fes)) return CB_ERR_ALIGN;
    }
    if (resid)
        for (int g = 0; g < ng; ++g)
            if (resid[g] && !aligned(resid[g], res)) return CB_ERR_ALIGN;
    int rc = check_gates(p, gates, gate_dtype);
    if (rc != CB_OK) return rc;
    if (p->has_last) {
        const double d = t - p->last_t;
        if (d == 0.0 || (p->dir != 0 && (d > 0 ? 1 : -1) != p->dir)) return CB_ERR_ORDER;
    }
    for (int j = 0; j < p->count; ++j)
        if (p->slot_t[(p->oldest() + j) % p->K] == t) return CB_ERR_NODES_DEGENERATE;

    // one-entry history of weight 1: the new features themselves
    Window one{};
    one.n = 1;
    const double w1[1] = {1.0};
    rc = run_launch(p, one, w1, nullptr, p->cache_dtype, resid, resid_dtype, stream, gates, gate_dtype, feats,
                    feat_dtype);
    if (rc != CB_OK) return rc;
    p->slot_t[p->next] = t;
    p->next = (p->next + 1) % p->K;
    if (p->count < p->K) ++p->count;
    p->has_last = true;
    p->last_t = t;
    return CB_OK;
}

int cb_weights(const cb_plan* p, double t_target, double* w_logical) {
    if (!p || !w_logical) return CB_ERR_ARG;
    const int n = live_entries(p);
    if (n == 0) return CB_ERR_HISTORY_NOT_FULL;
    return weights_for(p, live_window(p, n), t_target, w_logical);
}

int cb_taylor_weights(const double* node_t, int n, double t_target, double* w) {
    if (!node_t || !w || n < 1 || n > CB_MAX_K || !std::isfinite(t_target)) return CB_ERR_ARG;
    for (int i = 0; i < n; ++i)
        if (!std::isfinite(node_t[i])) return CB_ERR_ARG;
    double h = 1.0;
    if (n >= 2) {
        h = node_t[n - 1] - node_t[n - 2];
        if (h == 0.0) return CB_ERR_NODES_DEGENERATE;
        for (int i = 1; i < n; ++i)  // equispaced nodes only
            if (std::fabs((node_t[i] - node_t[i - 1]) - h) > 1e-9 * std::fabs(h)) return CB_ERR_ARG;
    }
    const double theta = n >= 2 ? (t_target - node_t[n - 1]) / h : 0.0;
    // f(t) ~ sum_i theta^i / i! nabla^i f_n, nabla^i f_n = sum_k (-1)^k C(i, k) f_{n-k}
    for (int j = 0; j < n; ++j) w[j] = 0.0;
    double pow_fact = 1.0;  // theta^i / i!
    for (int i = 0; i < n; ++i) {
        if (i > 0) pow_fact *= theta / i;
        double binom = 1.0;  // C(i, k)
        for (int k = 0; k <= i; ++k) {
            if (k > 0) binom = binom * (i - k + 1) / k;
            w[n - 1 - k] += pow_fact * ((k & 1) ? -binom : binom);
        }
    }
    return CB_OK;
}

int cb_plan_export_weights(const cb_plan* p, const double* targets, int n_targets, double* table) {
    if (!p || (n_targets > 0 && (!targets || !table)) || n_targets < 0) return CB_ERR_ARG;
    const int K = p->K, n = (int)p->node_t.size();
    for (int m = 0; m < n_targets; ++m) {
        const double t = targets[m];
        if (!std::isfinite(t)) return CB_ERR_ARG;
        // the K most recent nodes that precede t in sampling order
        int last = -1;
        for (int i = 0; i < n; ++i) {
            const double d = t - p->node_t[i];
            const bool before = p->dir >= 0 ? d > 0 : d < 0;
            if (before) last = i;
        }
        if (last + 1 < K) return CB_ERR_HISTORY_NOT_FULL;
        Window w{};
        w.n = K;
        for (int j = 0; j < K; ++j) {
            w.t[j] = p->node_t[last - K + 1 + j];
            w.tau[j] = p->node_tau[last - K + 1 + j];
        }
        const int rc = weights_for(p, w, t, &table[(size_t)m * K]);
        if (rc != CB_OK) return rc;
    }
    return CB_OK;
}

int cb_plan_history(const cb_plan* p, double* slot_t, int* head, int* count) {
    if (!p) return CB_ERR_ARG;
    if (slot_t)
        for (int j = 0; j < p->K; ++j) slot_t[j] = p->slot_t[j];
    if (head) *head = p->oldest();
    if (count) *count = p->count;
    return CB_OK;
}

int cb_plan_reset(cb_plan* p) {
    if (!p) return CB_ERR_ARG;
    p->next = p->count = 0;
    p->has_last = false;
    return CB_OK;
}

int cb_plan_set_option(cb_plan* p, int option, int64_t value) {
    if (!p) return CB_ERR_ARG;
    switch (option) {
    case CB_OPT_KERNEL:
        if (value != CB_KERNEL_AUTO && value != CB_KERNEL_DIRECT && value != CB_KERNEL_BULK) return CB_ERR_ARG;
        p->kernel = (int)value;
        return CB_OK;
    case CB_OPT_WAIT_NS:
        if (value < 0 || value > 60000000000LL) return CB_ERR_ARG;
        p->wait_ns = (unsigned long long)value;
        return CB_OK;
    case CB_OPT_PARTIAL_HISTORY:
        if (value != 0 && value != 1) return CB_ERR_ARG;
        p->partial = value != 0;
        return CB_OK;
    case CB_OPT_TEST_WITHHOLD:
        if (value != 0 && value != 1) return CB_ERR_ARG;
        p->withhold_first = (int)value;
        return CB_OK;
    default: return CB_ERR_ARG;
    }
}

int cb_plan_device_status(cb_plan* p, int* status, void* stream) {
    if (!p || !status) return CB_ERR_ARG;
    if (!p->cache) return CB_ERR_UNBOUND;
    if (!p->status_clear) {  // nothing has run since binding
        *status = 0;
        return CB_OK;
    }
    cudaStream_t s = (cudaStream_t)stream;
    int v = 0;
    cudaError_t e = cudaMemcpyAsync(&v, p->status_word(), sizeof(int), cudaMemcpyDeviceToHost, s);
    if (e == cudaSuccess) e = cudaMemsetAsync(p->status_word(), 0, sizeof(int), s);
    if (e == cudaSuccess) e = cudaStreamSynchronize(s);
    if (e != cudaSuccess) return cuda_fail(e, "device status");
    *status = v;
    return CB_OK;
}

int cb_plan_num_groups(const cb_plan* p) { return p ? (int)p->groups.size() : 0; }

void cb_plan_destroy(cb_plan* p) { delete p; }

const char* cb_status_string(int s) {
    switch (s) {
    case CB_OK: return "ok";
    case CB_ERR_ARG: return "invalid argument";
    case CB_ERR_ALIGN: return "misaligned pointer";
    case CB_ERR_NODES_DEGENERATE: return "duplicate node times (omega'(tau_j) = 0)";
    case CB_ERR_HISTORY_NOT_FULL: return "history buffer holds fewer than K entries";
    case CB_ERR_ORDER: return "pushed time does not continue the sampling direction";
    case CB_ERR_UNBOUND: return "no cache arena bound to the plan";
    case CB_ERR_CUDA: return "CUDA error";
    case CB_ERR_LIMIT: return "size limit exceeded";
    default: return "unknown status";
    }
}

const char* cb_last_error_message(void) { return g_last_error.c_str(); }

}  // extern "C"
