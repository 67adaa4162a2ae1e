/*
 * ecmoe.h -- C ABI of the GB300 expert-choice (EC) MoE layer, forward and backward.
 *
 * The layer (arXiv 2604.01622, Sec. 2.2 "Mixture-of-Experts Routing"):
 *   S = softmax_e(X Wr + br)                              router scores, S in R^{N x E}
 *   T_{e,g} = top-k_g tokens t of group g by S[t,e]        expert choice (Sec. 2.2), one group
 *                                                          per sequence (Sec. 5.2), per-sequence
 *                                                          capacity k_g (Sec. 4.2)
 *   Y_t = sum_{e: t in T_e} S[t,e] * FFN_e(x_t)            gated combine (Sec. 2.2); tokens no
 *                                                          expert picks get exactly 0
 *   FFN_e(x) = (silu(x Wg_e) * (x Wu_e)) Wd_e               SwiGLU experts (appendix
 *                                                          "Experimental Setup")
 * Ties in the top-k go to the lower token index; the tokens of one (expert, group)
 * are listed in ascending index. The backward pass treats the selection as fixed.
 *
 * Conventions shared by every call:
 *   - All arrays are row-major and contiguous. Device pointers unless stated.
 *   - dtype EC_F32: X, Y, dY, dX, Wr, Wg, Wu, Wd are float32.
 *     dtype EC_BF16: the same arrays are bf16 (raw 16-bit), accumulation is fp32.
 *     S, gates, br and every weight gradient are float32 in both modes.
 *   - Shapes: X, Y, dY, dX [N][d]; Wr [d][E]; br [E]; Wg, Wu [E][d][d_ff];
 *     Wd [E][d_ff][d]; S [E][N] (expert-major); idx, gate [E][M] with
 *     M = sum_g k_g: row e holds expert e's tokens, group g at offsets
 *     k_off[g] .. k_off[g+1]-1 where k_off is the prefix sum of k_g.
 *   - Device pointers must be 16-byte aligned. On the bf16 path d and d_ff must be
 *     multiples of 64.
 *   - Every compute call is asynchronous on `stream` (a cudaStream_t, NULL for the
 *     legacy default stream) and does no host synchronisation. Argument errors are
 *     returned before anything is launched. A kernel that gives up on a bounded
 *     wait records EC_ERR_TIMEOUT in a device status word; ec_check_device reads it.
 *   - The library never allocates device memory: the caller provides one workspace
 *     (ec_workspace_bytes) that holds the activations saved for the backward pass.
 *     The library never frees caller memory.
 *   - A context is not thread-safe; calls on one context must be ordered.
 */
#ifndef ECMOE_H
#define ECMOE_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  EC_OK = 0,
  EC_ERR_INVALID_ARG = 1, /* null pointer, misaligned pointer, bad enum */
  EC_ERR_SHAPE = 2,       /* inconsistent sizes, k_g outside [0, L_g], bad group offsets */
  EC_ERR_UNSUPPORTED = 3, /* valid but not implemented (e.g. bf16 with d % 64 != 0) */
  EC_ERR_CUDA = 4,        /* a CUDA runtime error; message in ec_last_error */
  EC_ERR_TIMEOUT = 5,     /* a device-side bounded wait expired (kernel returned early) */
  EC_ERR_WORKSPACE = 6,   /* workspace missing, too small or misaligned */
  EC_ERR_STATE = 7        /* call order violated (backward before forward, ...) */
} ec_status;

typedef enum { EC_F32 = 0, EC_BF16 = 1 } ec_dtype;

typedef struct ec_ctx ec_ctx;

/* Create a context for one layer shape.
 *   N tokens in G groups: group g holds tokens group_off[g] .. group_off[g+1]-1
 *   (host array of G+1 int32, group_off[0] = 0, non-decreasing, group_off[G] = N).
 *   k_g: host array of G int32 capacities, 0 <= k_g[g] <= group size (Sec. 4.2: the
 *   capacity may differ per sequence). M = sum k_g is the number of rows every expert
 *   processes (Sec. 2.2: each expert takes exactly its capacity).
 *   dtype: EC_F32 or EC_BF16.
 * Host arrays are copied; the caller keeps ownership. Returns EC_ERR_SHAPE on bad sizes. */
ec_status ec_ctx_create(ec_ctx** out, int32_t N, int32_t d, int32_t E, int32_t d_ff, int32_t G,
                        const int32_t* group_off, const int32_t* k_g, int32_t dtype);

/* Destroy a context (host memory only; the workspace stays the caller's). NULL is ignored. */
void ec_ctx_destroy(ec_ctx* ctx);

/* Replace the per-group capacities (Sec. 4.2: a new k_g per denoising step).
 * k_g: host array of G int32. sum(k_g) must not exceed the M the context was created with
 * (the workspace is sized for it); the context's M becomes sum(k_g). Synchronous: waits for
 * the whole device (no earlier kernel on any stream may still read the group tables), then
 * copies k_g to the device; call outside stream capture. Invalidates saved forward state. */
ec_status ec_ctx_set_capacity(ec_ctx* ctx, const int32_t* k_g);

/* The same update without a host round trip (Sec. 4.2: capacity that changes with the
 * masking ratio of every sequence, step after step). k_g_dev: device array of G int32,
 * read on `stream` by one small kernel, so a schedule computed on the device (or uploaded
 * ahead for many steps) takes effect in stream order with no copy and no synchronisation.
 * The new capacities must keep the context's current M: 0 <= k_g[g] <= L_g and
 * sum(k_g) == ec_rows_per_expert(ctx) (the FLOPs-matched schedules of Sec. 4.2 keep the
 * total; use ec_ctx_set_capacity to change it). The check runs on the device: if it fails,
 * the previous capacities stay in force and the next ec_check_device returns EC_ERR_SHAPE.
 * Needs the workspace; invalidates saved forward state. ec_ctx_set_workspace re-uploads the
 * capacities last given on the host. */
ec_status ec_ctx_set_capacity_async(ec_ctx* ctx, const int32_t* k_g_dev, void* stream);

/* Residual form for stacked layers x_{l+1} = x_l + EC(x_l) (off by default): with it on,
 * ec_moe_forward writes Y = X + EC(X) and ec_moe_backward writes dX = dY + (the input
 * gradient of EC), both fused into the combine and scatter kernels. Tokens no expert
 * picks then get Y_t = X_t. Invalidates saved forward state. */
ec_status ec_ctx_set_residual(ec_ctx* ctx, int32_t on);

/* Tile shapes of the tensor-core expert GEMMs (bf16 path; the fp32 path ignores it). An
 * implementation choice with no counterpart in the paper (the expert FFNs of Sec. 2.2 are
 * computed the same way under every policy). EC_TILES_AUTO (default) picks per GEMM: 256 x 512 output tiles per SM pair where the
 * output columns are a multiple of 512 and the GEMM's K loop is long enough (1024, or 2048
 * behind the gate/up epilogue) to hide the hand-over of their accumulator halves, else
 * 256 x 256. EC_TILES_256 always takes 256 x 256; EC_TILES_512 takes 256 x 512 wherever the
 * columns fill it. All three give bit-identical results (the same N = 256 MMAs run over K
 * in the same order, with the same epilogue arithmetic; only the tiling of the output
 * differs). Takes effect from the next call on the context; returns EC_ERR_INVALID_ARG for
 * any other value (the context keeps its policy). */
enum { EC_TILES_AUTO = 0, EC_TILES_256 = 1, EC_TILES_512 = 2 };
ec_status ec_ctx_set_tiles(ec_ctx* ctx, int32_t policy);

/* Current rows per expert M = sum k_g. */
int64_t ec_rows_per_expert(const ec_ctx* ctx);

/* Bytes of device workspace the context needs (saved activations, scores, selection,
 * backward scratch). Depends only on the creation-time sizes. */
size_t ec_workspace_bytes(const ec_ctx* ctx);

/* Attach a caller-owned device workspace of at least ec_workspace_bytes bytes, 256-byte
 * aligned. Uploads the group table with a synchronous copy; call outside stream capture.
 * The workspace must stay allocated while the context is used. */
ec_status ec_ctx_set_workspace(ec_ctx* ctx, void* workspace, size_t bytes);

/* Router and expert-choice selection only (Sec. 2.2).
 *   X [N][d], Wr [d][E] (dtype of the context), br [E] float or NULL.
 *   S_in: NULL to compute S from X and Wr; otherwise a float [E][N] score matrix to select
 *   from (X, Wr, br are then ignored and may be NULL).
 *   S_out: NULL or float [E][N], receives the scores used.
 *   idx [E][M] int32 and gate [E][M] float receive the selection (gate = S[idx, e]). */
ec_status ec_route(ec_ctx* ctx, const void* X, const void* Wr, const float* br,
                   const float* S_in, float* S_out, int32_t* idx, float* gate, void* stream);

/* Whole-layer forward (Sec. 2.2): Y [N][d] in the context's dtype. idx, gate, S_out as in
 * ec_route (each may be NULL). Saves what ec_moe_backward needs in the workspace, and
 * remembers the weight pointers, which must stay valid and unchanged until the backward
 * call. Wg, Wu [E][d][d_ff]; Wd [E][d_ff][d]. */
ec_status ec_moe_forward(ec_ctx* ctx, const void* X, const void* Wr, const float* br,
                         const void* Wg, const void* Wu, const void* Wd, void* Y,
                         int32_t* idx, float* gate, float* S_out, void* stream);

/* Backward of the last ec_moe_forward on this context: gradients of <dY, Y>.
 *   dY, dX [N][d] in the context's dtype (dX is overwritten).
 *   dWr [d][E], dbr [E] (NULL allowed), dWg, dWu [E][d][d_ff], dWd [E][d_ff][d]: float32,
 *   overwritten (not accumulated). The selection is held fixed; the gate gradient flows
 *   through the softmax Jacobian into dX and dWr. */
ec_status ec_moe_backward(ec_ctx* ctx, const void* dY, void* dX, float* dWr, float* dbr,
                          float* dWg, float* dWu, float* dWd, void* stream);

/* Shared experts (the paper's MoE block also has shared experts that process every token,
 * appendix "Token Coverage"; 2 per layer in its models, appendix "Experimental Setup").
 * S shared SwiGLU experts of width f each sum to one SwiGLU FFN of width d_ff_shared = S*f:
 * their weights are passed concatenated, Wg_s, Wu_s [d][d_ff_shared] (expert s in columns
 * s*f .. s*f+f-1) and Wd_s [d_ff_shared][d] (its rows), and their gradients come back in the
 * same layouts (float32). ec_ctx_set_shared must be called before ec_ctx_set_workspace
 * (it changes ec_workspace_bytes); 0 removes them. On the bf16 path d_ff_shared must be a
 * multiple of 64. With shared experts configured the layer is
 *   Y = FFN_shared(X) + [routed expert-choice output as in ec_moe_forward] (+ X if residual)
 * and ec_moe_forward / ec_moe_backward return EC_ERR_STATE: use the _shared calls. */
ec_status ec_ctx_set_shared(ec_ctx* ctx, int32_t d_ff_shared);
ec_status ec_moe_forward_shared(ec_ctx* ctx, const void* X, const void* Wr, const float* br,
                                const void* Wg, const void* Wu, const void* Wd, const void* Wg_s,
                                const void* Wu_s, const void* Wd_s, void* Y, int32_t* idx,
                                float* gate, float* S_out, void* stream);
ec_status ec_moe_backward_shared(ec_ctx* ctx, const void* dY, void* dX, float* dWr, float* dbr,
                                 float* dWg, float* dWu, float* dWd, float* dWg_s, float* dWu_s,
                                 float* dWd_s, void* stream);

/* Token choice (TC), the routing the paper compares expert choice against (Sec. 2.2,
 * "Token-choice"): every token t takes its k best experts E_t = TopK_e(S[t,e], k) and
 *   Y_t = sum_{e in E_t, pair kept} g[t,e] FFN_e(x_t),  g[t,e] = S[t,e] / sum_{e' in E_t} S[t,e']
 * (gates renormalised over the k chosen experts). With capacity >= 0 each expert keeps at
 * most `capacity` tokens, the first ones in ascending token order, and drops the rest (a
 * dropped pair contributes nothing; the token's other gates are unchanged); the paper's
 * capacity is ceil(CF k N / E) for a capacity factor CF. capacity < 0: dropless (no cap).
 * Ties in TopK go to the lower expert index; each token's choices are listed best first.
 * The backward pass holds the choices and drops fixed and differentiates through the gate
 * normalisation and the softmax.
 *
 * ec_tc_ctx_create makes a token-choice context (bf16 only: dtype must be EC_BF16, else
 * EC_ERR_UNSUPPORTED; 1 <= k <= min(E, 32)). Its workspace holds every expert's rows in one
 * tensor, each expert's region padded to a multiple of 256 rows (at most N k + 255 E rows).
 * On such a context ec_route, ec_moe_forward(_shared), ec_moe_backward(_shared),
 * ec_ctx_set_capacity and ec_ctx_set_shared return EC_ERR_STATE; ec_ctx_set_residual,
 * profiling, ec_check_device and the workspace calls work as for expert choice.
 *
 * ec_tc_forward: X, Wr, br, Wg, Wu, Wd, Y as in ec_moe_forward. Optional outputs (device,
 * NULL to skip): choice [N][k] int32 expert ids best first, gate [N][k] float normalised
 * gates, kept [N][k] int32 (1 kept, 0 dropped), load [E] int32 tokens kept per expert,
 * S_out [N][E] float router scores (token-major, unlike the expert-choice calls).
 * ec_tc_backward: arguments as in ec_moe_backward; needs a preceding ec_tc_forward on the
 * same context whose inputs are still alive. */
ec_status ec_tc_ctx_create(ec_ctx** out, int32_t N, int32_t d, int32_t E, int32_t d_ff,
                           int32_t k, int32_t capacity, int32_t dtype);

/* Token-choice expert capacity for a capacity factor (Sec. 2.2): ceil(CF k N / E), evaluated
 * left to right in double precision, for the `capacity` argument of ec_tc_ctx_create.
 * Returns -1 (dropless, no cap) for capacity_factor <= 0 or NaN, -2 for k < 1, N < 0,
 * E < 1 or a result that does not fit. Host only. */
int64_t ec_tc_capacity(double capacity_factor, int32_t k, int32_t N, int32_t E);
ec_status ec_tc_forward(ec_ctx* ctx, const void* X, const void* Wr, const float* br,
                        const void* Wg, const void* Wu, const void* Wd, void* Y, int32_t* choice,
                        float* gate, int32_t* kept, int32_t* load, float* S_out, void* stream);
ec_status ec_tc_backward(ec_ctx* ctx, const void* dY, void* dX, float* dWr, float* dbr,
                         float* dWg, float* dWu, float* dWd, void* stream);

/* Synchronise `stream`, read and clear the device status word. Returns EC_ERR_TIMEOUT if a
 * kernel gave up on a bounded wait since the last check, EC_ERR_SHAPE if a capacity update
 * from device memory (ec_ctx_set_capacity_async) was rejected, EC_ERR_CUDA on a CUDA error. */
ec_status ec_check_device(ec_ctx* ctx, void* stream);

/* Per-kernel timing. With profiling on, every kernel launch of the following calls is
 * bracketed by CUDA events recorded on the call's stream (one event record per kernel;
 * off by default). Phases accumulate over calls; ec_ctx_set_profiling clears them. */
ec_status ec_ctx_set_profiling(ec_ctx* ctx, int32_t on);

/* Phases recorded since profiling was last switched: up to `cap` kernel names (static
 * strings) and durations in ms, in launch order. Waits for the last recorded event.
 * Returns the number of phases (which may exceed cap), 0 if none, -1 on a CUDA error. */
int32_t ec_ctx_profile(ec_ctx* ctx, const char** names, float* ms, int32_t cap);

/* Number of CUDA kernels the library has launched through this context so far. */
int64_t ec_kernel_launches(const ec_ctx* ctx);

/* Capacity schedulers (Sec. 4.2, Table 1): masking ratio r -> top-k equivalent
 *   k(r) = clamp(k_min + (k_max - k_min) s(r), k_min, k_max) with
 *   s = 1/2 (static), r, 1 - r, (1 - cos pi r)/2, (1 + cos pi r)/2, g~(r), 1 - g~(r), where
 *   g~(r) = (g(r) - g(0)) / (1 - g(0)), g(r) = exp(-(r - 1/2)^2 / (2 sigma^2)) (appendix
 *   "Scheduler Definitions and FLOPs Equivalence"; the paper uses sigma = 0.22). */
typedef enum {
  EC_SCHED_STATIC = 0,
  EC_SCHED_LINEAR = 1,
  EC_SCHED_LINEAR_REV = 2,
  EC_SCHED_COSINE = 3,
  EC_SCHED_COSINE_REV = 4,
  EC_SCHED_GAUSSIAN = 5,
  EC_SCHED_GAUSSIAN_REV = 6
} ec_scheduler;

/* Per-sequence capacities for one step (host only, no GPU needed): group g has masking ratio
 * r[g] in [0, 1] and L_g = group_off[g+1] - group_off[g] tokens; expert capacity
 * k_g[g] = floor(k(r[g]) * L_g / E + 1/2) clipped to [0, L_g] (Sec. 2.2: c = k N / E per
 * selection pool). Host arrays: group_off [G+1], r [G], k_g [G] (written). sigma is used by
 * the Gaussian schedulers only. EC_ERR_INVALID_ARG on an unknown scheduler, r outside
 * [0, 1], k_min < 0 or k_max < k_min; EC_ERR_SHAPE on bad sizes. The result feeds
 * ec_ctx_set_capacity (whose sum(k_g) limit is the caller's to respect). */
ec_status ec_capacity_schedule(int32_t scheduler, double k_min, double k_max, double sigma,
                               int32_t E, int32_t G, const int32_t* group_off, const double* r,
                               int32_t* k_g);

/* Failure-path self-test (no counterpart in the paper): launches one kernel that waits on
 * an mbarrier that nothing completes, with the same bounded wait the tensor-core kernels
 * use but a limit of limit_ns nanoseconds (at most 10 s). The kernel gives up, records the
 * timeout in the context's device status word and returns, so the context stays usable;
 * ec_check_device then reports EC_ERR_TIMEOUT once. Asynchronous on `stream`. */
ec_status ec_selftest_bounded_wait(ec_ctx* ctx, uint64_t limit_ns, void* stream);

/* Expert-choice selection for callers that cannot allocate device memory (the paper has no
 * counterpart: this is a deployment variant of the selection in ec_route).
 *
 * Some callers cannot call cudaMalloc where they need a selection: a runtime that hands
 * out a fixed memory budget, or code that must not grow the device footprint once it is
 * serving. This call needs no context and no workspace: its scratch (the token->slot map
 * and the group tables) lives in one file-scope device array of
 * EC_STATIC_SELECT_MAX_SCORES + 3*(EC_STATIC_SELECT_MAX_GROUPS+1) int32 (about 16 MB), which
 * every GPU that loads the library holds until the process exits. It calls no allocator.
 *   S [E][N] float scores (device), N tokens in G groups given by the host arrays
 *   group_off [G+1] and k_g [G] (same rules as ec_ctx_create); idx [E][M] int32 and
 *   gate [E][M] float (device, M = sum k_g) receive the same selection as ec_route with S_in.
 * Returns EC_ERR_UNSUPPORTED if N*E > EC_STATIC_SELECT_MAX_SCORES or
 * G > EC_STATIC_SELECT_MAX_GROUPS, EC_ERR_SHAPE / EC_ERR_INVALID_ARG on bad arguments,
 * EC_ERR_CUDA if a CUDA call fails. Asynchronous on `stream`. The call copies group_off and
 * k_g into its own host array before it enqueues anything, so the caller may reuse or free
 * them (pinned or pageable) as soon as it returns. It returns EC_ERR_UNSUPPORTED, having
 * enqueued nothing, while `stream` is being captured: the group tables are copied from host
 * memory that lives only for the duration of the call. The first call in each CUDA context
 * (a device's primary context, and again after cudaDeviceReset) looks up the array's device
 * address; make that first call before any stream capture. All calls share the array:
 * calls that overlap on the GPU (other streams, other threads) race and must be ordered. */
#define EC_STATIC_SELECT_MAX_SCORES 4194304
#define EC_STATIC_SELECT_MAX_GROUPS 4096
ec_status ec_select_static(const float* S, int32_t N, int32_t E, int32_t G,
                           const int32_t* group_off, const int32_t* k_g, int32_t* idx,
                           float* gate, void* stream);

/* Message of the last failed call on this context ("" if none). Owned by the context. */
const char* ec_last_error(const ec_ctx* ctx);

/* The same message copied into a caller buffer: at most n-1 bytes and a terminating NUL
 * (nothing is written when n is 0). Returns the status of the last failed call on the
 * context (EC_OK if none has failed), or EC_ERR_INVALID_ARG for a NULL context, or a NULL
 * buffer with n > 0. Device-side failures reach the message through ec_check_device. */
ec_status ec_get_last_error(const ec_ctx* ctx, char* buf, size_t n);

/* Static name of a status code. */
const char* ec_status_string(ec_status s);

#ifdef __cplusplus
}
#endif
#endif /* ECMOE_H */
