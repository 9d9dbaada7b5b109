/*
 * chebboost.h — C ABI of libchebboost, a GB300 (sm_103a) implementation of the
 * online extrapolation stage of ChebBooster (training-free DiT acceleration by
 * Chebyshev-inspired barycentric extrapolation).
 *
 * The method (paper Sec. 3.2-3.3, Alg. 1):
 *   - on full-computation steps s in F, every block's branch outputs f_s are
 *     stored in a history buffer H that holds the n = K most recent
 *     (s_j, f_j) pairs, dropping the oldest (Sec. 3.3, the forward
 *     application; Alg. 1, full-computation branch);
 *   - on every other step t the features are predicted as
 *         f_t = sum_j w^j_t f_{s_j}                       (Sec. 3.3, Eq. for f_t)
 *     with the barycentric interpolation coefficients
 *         w^j_t = (rho_j / (tau - tau_j)) / sum_i rho_i / (tau - tau_i)
 *                                                  (Sec. 3.2, Eq. barycentric_coeff)
 *     where rho_j = 1 / prod_{k != j} (tau_j - tau_k)   (App. A, Eq. general_weights)
 *     and tau is the timestep mapped affinely onto [-1, 1] (Sec. 3.3).
 *
 * Conventions for every call:
 *   - Host/device: "device pointer" means memory the current CUDA device's
 *     kernels can address: its own memory, or host memory mapped into the
 *     device's address space (pinned, UVA-mapped buffers, which the kernels
 *     then read or write over the CPU-GPU link). "host pointer" means ordinary
 *     process memory read by the host code. The plan holds host state only;
 *     the caller owns and allocates every buffer (cache arena, features,
 *     outputs, hidden states) and every stream.
 *   - Streams: `stream` is a cudaStream_t passed as void* (NULL = the legacy
 *     default stream). Device work is enqueued on it asynchronously; no call
 *     synchronises the device.
 *   - Errors: every call validates all of its arguments before enqueueing
 *     anything. On a negative status nothing was enqueued and the plan's
 *     state (its history) is unchanged. CB_ERR_CUDA reports a failed launch;
 *     cb_last_error_message() gives the CUDA error text.
 *   - Threads: a plan is not internally locked; calls on the same plan must
 *     be serialised by the caller. Different plans are independent.
 *   - Layout: each branch tensor is a contiguous row-major array
 *     [batch, tokens, hidden] of `numel` elements. Pointers must be aligned to
 *     their element size; pointers aligned to 16 bytes take the vectorised
 *     path, others a scalar path (same results).
 *   - Rounding: fp32 -> bf16 conversions round to nearest, ties to even.
 */
#ifndef CHEBBOOST_H
#define CHEBBOOST_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define CB_MAX_K 8            /* largest history size n (Sec. 3.3) */
#define CB_MAX_TENSORS 256    /* branch tensors per plan */
#define CB_MAX_BRANCHES 4     /* branch tensors sharing one residual group */
#define CB_MAX_NUMEL (1LL << 48) /* elements per branch tensor */
#define CB_CACHE_ALIGN 256    /* byte alignment of the cache arena and of each tensor in it */
#define CB_STATUS_BYTES 256   /* device status block at the end of the cache arena */

typedef struct cb_plan cb_plan; /* opaque, host-owned */

typedef enum { CB_BF16 = 0, CB_FP32 = 1 } cb_dtype;

/* One cached branch tensor (Sec. 3.1: the self-attention, cross-attention
 * and MLP outputs S^l, C^l, M^l of block l). `group` names the hidden state
 * the branch is added into (B^l(x) = x + S^l + C^l + M^l): tensors with the
 * same group share one residual pointer in cb_extrapolate and must have the
 * same numel; -1 means the tensor has no residual. */
typedef struct {
    int32_t layer;    /* block index l (informational) */
    int32_t branch;   /* branch index inside the block (informational) */
    int64_t numel;    /* elements = batch * tokens * hidden, > 0 */
    int32_t group;    /* residual group in [0, n_groups) or -1 */
    int32_t reserved; /* must be 0 */
} cb_tensor_desc;

enum {
    CB_OK = 0,
    CB_ERR_ARG = -1,               /* null, out-of-range or inconsistent argument */
    CB_ERR_ALIGN = -2,             /* pointer not aligned to its element size (cache: 256 B) */
    CB_ERR_NODES_DEGENERATE = -3,  /* duplicate node times: omega'(tau_j) = 0 (App. A) */
    CB_ERR_HISTORY_NOT_FULL = -4,  /* fewer than K entries in H (Sec. 3.3 requires |H| = n) */
    CB_ERR_ORDER = -5,             /* pushed time does not continue the sampling direction */
    CB_ERR_UNBOUND = -6,           /* no cache arena bound to the plan */
    CB_ERR_CUDA = -7,              /* a CUDA call or launch failed */
    CB_ERR_LIMIT = -8              /* a size beyond one of the CB_MAX_* limits */
};

/* Options of cb_plan_set_option. */
enum {
    CB_OPT_KERNEL = 1,  /* skipped-step kernel: CB_KERNEL_AUTO (default), _DIRECT or _BULK */
    CB_OPT_WAIT_NS = 2, /* limit of every device-side wait of the bulk kernel, ns
                           (default 1e9, at most 6e10) */
    CB_OPT_TEST_WITHHOLD = 3, /* 1: (tests of the failure path only) the bulk kernel's producer
                                 announces each CTA's first unit but never issues its copies, so
                                 that the consumers' wait runs out; outputs are then invalid */
    CB_OPT_PARTIAL_HISTORY = 4 /* 1: while H holds m < K entries (m >= 1), skipped steps use those m
                                  (degree m-1 extrapolation; m = 1 reuses the newest features)
                                  instead of failing with CB_ERR_HISTORY_NOT_FULL. This is Alg. 1
                                  read literally (extrapolate from whatever H holds); default 0,
                                  the text's reading (extrapolate only once |H| = n) */
};
enum { CB_KERNEL_AUTO = 0, CB_KERNEL_DIRECT = 1, CB_KERNEL_BULK = 2 };

/* Codes OR-ed into the device status word (cb_plan_device_status). */
enum {
    CB_DEV_CONSUMER_TIMEOUT = 1, /* a consumer's wait for a filled stage ran out */
    CB_DEV_PRODUCER_TIMEOUT = 2, /* the producer's wait for a released stage ran out */
    CB_DEV_DRAIN_TIMEOUT = 4     /* the producer's final wait for its own copies ran out */
};

/* Full-computation schedule (Sec. 3.3, Eq. for F; Alg. 1 offline stage):
 *   s in F  iff  s not in [s0, T-1-s1]  or  r divides (s - s0),   s in [0, T-1],
 * then, when K > 0, every step whose history would hold fewer than K entries
 * is also marked full (Sec. 3.3 extrapolates only once H holds n entries).
 * is_full: host array of T bytes, written 1 (full) or 0 (extrapolated).
 * n_full: host int, receives the number of full steps (may be NULL).
 * Errors: CB_ERR_ARG for T <= 0, r <= 0, s0 < 0, s1 < 0, K < 0 or is_full NULL. */
int cb_schedule_full(int T, int r, int s0, int s1, int K, uint8_t* is_full, int* n_full);

/* Offline precomputation (the weight precomputation of Sec. 3.3; Alg. 1, offline
 * stage). node_t: host array of the n_nodes timesteps at which full
 * computations happen, in sampling order (strictly monotone). For every
 * window of K consecutive nodes the fp64 barycentric weights rho_j of
 * App. A, Eq. general_weights, are computed here on the normalised times
 * tau = 2 (t - t_min) / (t_max - t_min) - 1. tensors: host array of n_tensors
 * descriptors (copied). cache_dtype: storage type of the history buffer.
 * out: receives the new plan. Errors: CB_ERR_ARG (K < 1, n_nodes < K, bad
 * descriptor, t_min >= t_max, non-monotone nodes), CB_ERR_LIMIT (K >
 * CB_MAX_K, more than CB_MAX_TENSORS tensors or CB_MAX_BRANCHES members of
 * a group, a group index >= CB_MAX_TENSORS, numel > CB_MAX_NUMEL),
 * CB_ERR_NODES_DEGENERATE (repeated node time). */
int cb_plan_create(const double* node_t, int n_nodes, int K, const cb_tensor_desc* tensors,
                   int n_tensors, cb_dtype cache_dtype, double t_min, double t_max, cb_plan** out);

/* Bytes of device memory the history buffer needs: K slots followed by a
 * CB_STATUS_BYTES status block. Slot p starts at p * slot_bytes; inside it
 * tensor i starts at sum_{k<i} roundup(numel_k * esize, CB_CACHE_ALIGN). */
size_t cb_plan_cache_bytes(const cb_plan* plan);

/* Attach caller-owned device memory as the history buffer (the plan never
 * allocates device memory). dev_ptr must be CB_CACHE_ALIGN-aligned and
 * bytes >= cb_plan_cache_bytes. Rebinding empties the history.
 * Errors: CB_ERR_ARG, CB_ERR_ALIGN. */
int cb_plan_bind_cache(cb_plan* plan, void* dev_ptr, size_t bytes);

/* Full step (Sec. 3.3; Alg. 1, full-computation branch): store the pair
 * (t, f_t) in H. feats: host array of n_tensors device pointers, one per
 * tensor descriptor, each numel elements of feat_dtype. One grouped kernel
 * writes every tensor into the ring slot that holds the oldest entry (or the
 * next free slot), converting fp32 -> bf16 (RNE) when the cache is bf16
 * (bf16 -> bf16 is a bit copy, bf16 -> fp32 exact). t must continue the
 * sampling direction of node_t strictly (CB_ERR_ORDER otherwise).
 * Errors: CB_ERR_ARG, CB_ERR_ALIGN, CB_ERR_UNBOUND, CB_ERR_ORDER, CB_ERR_CUDA. */
int cb_cache_push(cb_plan* plan, const void* const* feats, cb_dtype feat_dtype, double t, void* stream);

/* Skipped step (Sec. 3.3, Eq. for f_t; Alg. 1, extrapolation branch): for
 * every tensor i and element e,
 *     P_i[e] = sum_j w_j(t_target) F_{i,j}[e]
 * over the K entries of H, with the fp64 weights of Eq. barycentric_coeff
 * computed on the host from the live node times. The weights travel as kernel
 * parameters (an fp32 high/low pair each); one grouped persistent kernel
 * covers all tensors, accumulating in fp32 with a compensated fallback, so
 * that bf16 results are within one bf16 ulp of the exactly rounded value.
 * outs: host array of n_tensors device pointers (entries may be NULL; the
 *       array itself may be NULL), each receiving P_i as out_dtype.
 * resid: host array of n_groups device pointers (may be NULL; entries may be
 *       NULL). For group g, resid[g] <- round(resid[g] + sum_{i in g} P_i)
 *       in place, with one rounding to resid_dtype (the block residual of
 *       Sec. 3.1 with cached branches).
 * A target equal to a node time returns that node's features exactly.
 * Errors: CB_ERR_ARG, CB_ERR_ALIGN, CB_ERR_UNBOUND, CB_ERR_HISTORY_NOT_FULL,
 * CB_ERR_CUDA. */
int cb_extrapolate(cb_plan* plan, double t_target, void* const* outs, cb_dtype out_dtype,
                   void* const* resid, cb_dtype resid_dtype, void* stream);

/* As cb_extrapolate, for a history described by the caller (Sec. 3.3: H
 * holds the n most recent pairs and the oldest is discarded, so a ring buffer
 * holds them in rotated order). slot_t: host array of K times, slot_t[p]
 * being the timestep whose features ring slot p holds; head: the slot of the
 * OLDEST entry (logical order head, head+1, ... mod K). No data moves: only
 * the weights are permuted to slot order. The plan's own history must be
 * full (every slot written). Errors: as cb_extrapolate, plus
 * CB_ERR_NODES_DEGENERATE for repeated slot times. */
int cb_extrapolate_ring(cb_plan* plan, const double* slot_t, int head, double t_target,
                        void* const* outs, cb_dtype out_dtype, void* const* resid,
                        cb_dtype resid_dtype, void* stream);

/* The skipped step of cb_extrapolate_ring for callers that may not allocate
 * device memory. The paper has no counterpart: this is a library convenience.
 * Who needs it: an operator running inside a framework or inference engine
 * that lays out every device buffer ahead of time. Such an operator is handed
 * its input and output buffers and must not call cudaMalloc. The same holds
 * for a process whose memory pool has already reserved the GPU. Such a caller
 * can hold the history in a buffer of exactly K slots, but it cannot add the
 * CB_STATUS_BYTES status block that cb_plan_bind_cache asks for. This call
 * needs neither: the plan need not be bound, and the kernel records its
 * device-side events in a block the library holds itself.
 *
 * plan: a plan from cb_plan_create. Only its tensor descriptors, K, time
 *       interval, node table and options are used: its own history is
 *       neither read nor changed.
 * hist: device pointer to the caller's history buffer, CB_CACHE_ALIGN-aligned,
 *       laid out like the arena's first K slots (slot p at p * slot_bytes,
 *       slot_bytes = (cb_plan_cache_bytes(plan) - CB_STATUS_BYTES) / K).
 *       hist_bytes: its size, at least K * slot_bytes.
 * slot_t, head, t_target, outs, out_dtype, resid, resid_dtype, stream:
 *       as cb_extrapolate_ring. Every slot must hold an entry.
 * status: host pointer (may be NULL). It receives the launch's device status
 *       word (CB_DEV_* codes, 0 = none) once the stream has reached the end
 *       of this call. The value arrives by an asynchronous device-to-host
 *       copy when *status is pinned memory. With ordinary memory the copy,
 *       and thus this call, waits for the launch to finish.
 *
 * Allocation: the call allocates no device memory and no pinned host memory.
 * Its status block is a file-scope device array of CB_STATUS_BYTES (256) bytes. Every GPU that
 * loads the library holds it until the process exits. A call uses one 4-byte
 * word of it whatever the workload's size, so no workload can outgrow it. The
 * call still rejects a history buffer smaller than the K slots (CB_ERR_ARG),
 * sizes beyond the CB_MAX_* limits and device ordinals from 64 up
 * (CB_ERR_LIMIT).
 * Set-up: the first call on each device looks up the block's device address
 * there (cudaGetSymbolAddress, with that device current). Make that first call
 * before any stream capture begins.
 * Sharing: every call on a device uses the same word. Each launch clears it
 * first on its own stream. Calls that overlap on the GPU (different streams,
 * no ordering between them) race on it: one may clear or read another's
 * code. Their outputs are unaffected.
 * Errors: as cb_extrapolate_ring (CB_ERR_UNBOUND excepted), plus CB_ERR_ALIGN
 * for hist and CB_ERR_CUDA when the status block cannot be reached. A
 * CB_ERR_CUDA from the status read-back comes after the launch was enqueued. */
int cb_extrapolate_noalloc(cb_plan* plan, const void* hist, size_t hist_bytes, const double* slot_t,
                           int head, double t_target, void* const* outs, cb_dtype out_dtype,
                           void* const* resid, cb_dtype resid_dtype, int* status, void* stream);

/* Shapes of the branch tensors, needed by the gated calls: bth[3*i + 0..2] =
 * batch, tokens, hidden of tensor i (their product must be its numel;
 * tokens * hidden < 2^32). Tensors of one residual group must share tokens
 * and hidden. Errors: CB_ERR_ARG, CB_ERR_LIMIT. */
int cb_plan_set_shapes(cb_plan* plan, const int64_t* bth);

/* Skipped step with gated hidden-state updates. DiT blocks add each branch
 * through a per-sample, per-channel gate computed from the timestep
 * conditioning (the adaptive normalisation of the blocks, Sec. 3.1); when the
 * cache holds the un-gated branch outputs, the gate of the current step
 * multiplies the prediction:
 *     resid[g] <- round(resid[g] + sum_{i in g} gate_i[b, h] * P_i[b, tok, h]).
 * gates: host array of n_tensors pointers (NULL array or entries: gate 1),
 * each a [batch, hidden] array of gate_dtype broadcast over tokens; shapes
 * must be set (cb_plan_set_shapes). Predictions written to outs stay
 * un-gated. Otherwise as cb_extrapolate; errors as cb_extrapolate. */
int cb_extrapolate_gated(cb_plan* plan, double t_target, void* const* outs, cb_dtype out_dtype,
                         void* const* resid, cb_dtype resid_dtype, const void* const* gates,
                         cb_dtype gate_dtype, void* stream);

/* Full step with its epilogue fused (Sec. 3.3 / Alg. 1, full-computation
 * branch, plus the block residual of Sec. 3.1): one pass stores every branch
 * output in H exactly as cb_cache_push does and, for each residual group g
 * with resid[g] non-NULL, adds the un-rounded outputs into the hidden state:
 *     resid[g] <- round(resid[g] + sum_{i in g} gate_i * feats_i)
 * (one rounding of the un-rounded sum, with the accuracy of cb_extrapolate's
 * hidden-state update; gates as in cb_extrapolate_gated, may be NULL). It runs
 * the skipped-step kernels on a one-entry history of weight 1 (the features
 * themselves), so it saves the separate read of the features that the
 * residual add would otherwise need. Errors: as cb_cache_push, plus those of
 * the gates. */
int cb_cache_push_residual(cb_plan* plan, const void* const* feats, cb_dtype feat_dtype, double t,
                           void* const* resid, cb_dtype resid_dtype, const void* const* gates,
                           cb_dtype gate_dtype, void* stream);

/* Skipped step with caller-chosen weights: P_i = sum_j w_logical[j] F_{i,j}
 * over the live history (the kernel of cb_extrapolate with the weights of
 * Sec. 3.3's linear combination given directly, e.g. another node family's
 * coefficients or finite-difference Taylor weights, see cb_taylor_weights).
 * w_logical: host array of n doubles, oldest .. newest, n = K (or the number of
 * live entries under CB_OPT_PARTIAL_HISTORY); outs, resid and errors as
 * cb_extrapolate (non-finite weights: CB_ERR_ARG). */
int cb_extrapolate_weights(cb_plan* plan, const double* w_logical, void* const* outs, cb_dtype out_dtype,
                           void* const* resid, cb_dtype resid_dtype, void* stream);

/* The fp64 weights cb_extrapolate would use for t_target on the live history
 * (Eq. barycentric_coeff), in logical order oldest .. newest. w_logical: host
 * array of n doubles, n = K (or the number of live entries under
 * CB_OPT_PARTIAL_HISTORY). Errors: CB_ERR_ARG, CB_ERR_HISTORY_NOT_FULL. */
int cb_weights(const cb_plan* plan, double t_target, double* w_logical);

/* The precomputed weight table (Sec. 3.3; Alg. 1, offline stage): for each
 * targets[m] the weights over the K most recent nodes of node_t that precede
 * it in sampling order, written to table[m*K + j] (j oldest .. newest).
 * Errors: CB_ERR_ARG, CB_ERR_HISTORY_NOT_FULL (fewer than K nodes precede a
 * target). */
int cb_plan_export_weights(const cb_plan* plan, const double* targets, int n_targets, double* table);

/* Truncated-Taylor extrapolation weights (the Taylor expansion the paper
 * compares against in Sec. 3.2, Fig. 4), with derivatives estimated by
 * backward differences on n equispaced nodes: with h the node spacing and
 * theta = (t_target - node_t[n-1]) / h,
 *     f(t_target) ~ sum_{i<n} theta^i / i! * nabla^i f(node_t[n-1]),
 *     nabla^i f_n = sum_{k<=i} (-1)^k C(i, k) f_{n-k}.
 * w: host array of n doubles (oldest .. newest) for cb_extrapolate_weights.
 * n = 1 gives w = (1): reuse of the newest features. Errors: CB_ERR_ARG (n out
 * of [1, CB_MAX_K], nodes not equispaced), CB_ERR_NODES_DEGENERATE. */
int cb_taylor_weights(const double* node_t, int n, double t_target, double* w);

/* Introspection of H: slot_t (host, K doubles) receives each slot's time,
 * head the slot of the oldest entry, count the number of entries (<= K).
 * Any output pointer may be NULL. */
int cb_plan_history(const cb_plan* plan, double* slot_t, int* head, int* count);

/* Set a plan option (CB_OPT_*). CB_OPT_KERNEL selects the skipped-step
 * kernel: the direct-load kernel (each thread loads its K vectors from HBM) or
 * the bulk-copy pipeline (a producer warp stages the K chunks of each tile in
 * shared memory with cp.async.bulk; a persistent grid of one or two CTAs per
 * SM); both compute identical bits. CB_OPT_WAIT_NS bounds every wait of the bulk kernel
 * on a shared-memory barrier; a wait that runs out makes the kernel record a
 * CB_DEV_* code in the device status word and return early (its outputs are
 * then incomplete). Errors: CB_ERR_ARG. */
int cb_plan_set_option(cb_plan* plan, int option, int64_t value);

/* Read the device status word into *status (0 = no device-side event since
 * the last read) and clear it. Enqueues a 4-byte copy and a 4-byte memset on
 * `stream` and synchronises that stream. Errors: CB_ERR_ARG, CB_ERR_UNBOUND,
 * CB_ERR_CUDA. */
int cb_plan_device_status(cb_plan* plan, int* status, void* stream);

/* Empty H (a new sample starts). */
int cb_plan_reset(cb_plan* plan);

/* Number of residual groups (1 + the largest descriptor group, 0 if none). */
int cb_plan_num_groups(const cb_plan* plan);

void cb_plan_destroy(cb_plan* plan);

/* Static text for a status code. */
const char* cb_status_string(int status);

/* Text of the most recent CB_ERR_CUDA on the calling thread ("" if none). */
const char* cb_last_error_message(void);

#ifdef __cplusplus
}
#endif

#endif /* CHEBBOOST_H */
