/*
 * unif_moe.h - C ABI of the GB300 (sm_103a) UniF-MoE layer forward pass.
 *
 * The layer ("Share First, Route What Remains", Sec. III) holds one shared
 * expert and K residual experts, each an FFN of width H = d_ff split into B
 * aligned blocks of width M = H / B (Sec. III-A, Eq. 16). For every token x:
 *   alpha = tau + (1 - 2 tau) sigmoid(x W_shr), tau = (B-1)/B^2    (Eq. 18)
 *   b     = round(B alpha) shared blocks                          (Eq. 19)
 *   I_shr = the b blocks of largest priority u_b = x mu_b, where
 *           mu_b is the mean of the shared keys of block b         (Eqs. 20-23)
 *   s     = softmax(x W_g) over the K residual experts, sorted as
 *           p_1 >= ... >= p_K with experts q_1..q_K                (Eqs. 24-25)
 *   k     = smallest n with p_1 + ... + p_n >= beta = 1 - alpha    (Eqs. 26-27)
 *   y     = alpha * sum_{b in I_shr} E_shr^(b)(x)
 *           + sum_{i<=k} p_i * sum_{b not in I_shr} E_{q_i}^(b)(x)   (Eqs. 28-30)
 * and it activates C_B = b + k (B - b) blocks (Eq. 35).
 *
 * Conventions for every call below:
 *   - Pointers named *_dev are device pointers; the caller owns them. Pointers
 *     named *_host are host pointers (pinned memory gives the fastest copies).
 *   - `stream` is a cudaStream_t (NULL = the legacy default stream). Work is
 *     enqueued on it; calls return without synchronising unless stated.
 *   - Return value: UNIF_MOE_OK (0) or a negative UNIF_MOE_ERR_* code; the
 *     message of the last failure on the calling thread is returned by
 *     unif_moe_last_error().
 *   - Rows are row-major and densely packed; element type is the layer dtype
 *     (float for UNIF_MOE_F32, bfloat16 for UNIF_MOE_BF16) unless stated.
 *   - Device pointers handed to unif_moe_forward must be 16-byte aligned.
 * A handle may be used from one host thread at a time; forwards on one
 * handle share its workspace, so they must be ordered on a single stream.
 */
#ifndef UNIF_MOE_H
#define UNIF_MOE_H

#include <stdint.h>

#if defined(__GNUC__)
#define UNIF_MOE_API __attribute__((visibility("default")))
#else
#define UNIF_MOE_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

typedef struct unif_moe_layer* unif_moe_t;

enum {
  UNIF_MOE_OK = 0,
  UNIF_MOE_ERR_ARG = -1,      /* null or misaligned pointer, value out of range */
  UNIF_MOE_ERR_SHAPE = -2,    /* layer shape the kernels do not support */
  UNIF_MOE_ERR_CAPACITY = -3, /* T larger than max_tokens of the handle */
  UNIF_MOE_ERR_CUDA = -4,     /* a CUDA runtime or driver call failed */
  UNIF_MOE_ERR_TIMEOUT = -5,  /* a kernel gave up waiting (see sync_status) */
  UNIF_MOE_ERR_STATE = -6     /* call out of order, e.g. forward before load */
};

typedef enum { UNIF_MOE_F32 = 0, UNIF_MOE_BF16 = 1 } unif_moe_dtype;

/* Routing thresholds. NaN / 0 select the paper's adaptive rule; the other
 * values are the non-adaptive replacements the paper ablates (Table IV). */
typedef struct {
  float tau;         /* NaN: (B-1)/B^2 (Eq. 18); else this tau */
  float alpha_fixed; /* NaN: adaptive alpha (Eq. 18); else this constant alpha,
                        which sets b (Eq. 19) and the shared weight */
  float beta_fixed;  /* NaN: beta = 1 - alpha (Eq. 26); else this constant
                        cumulative-mass threshold theta */
  int topk_fixed;    /* 0: cumulative count (Eq. 27); else k = topk_fixed */
  int prefix_blocks; /* 0: TopK of prototype priorities (Eq. 22); 1: the
                        first b blocks */
} unif_moe_thresholds;

/* Fills *th with the paper's adaptive settings (all NaN / 0). */
UNIF_MOE_API void unif_moe_default_thresholds(unif_moe_thresholds* th);

/* Optional parts of a handle, chosen at create time (not in the paper; they
 * decide which workspaces unif_moe_create_ex allocates up front). */
enum {
  UNIF_MOE_FEATURE_NORM_FIRST = 1, /* unif_moe_sublayer_forward with norm_first:
                                      a [max_tokens][d] buffer for LN(x) */
  UNIF_MOE_FEATURE_HOST_IO = 2,    /* unif_moe_forward_host(_async): two slots
                                      of device staging buffers for x, y, the
                                      mask and the counts, two copy streams */
  UNIF_MOE_FEATURE_BACKWARD = 4,   /* unif_moe_backward: transposed copies of the
                                      expert weights and per-row gradient buffers
                                      (bf16 layers, d % 128 == 0) */
  UNIF_MOE_FEATURE_DIAGNOSTICS = 8, /* unif_moe_value_alignment and
                                      unif_moe_functional_demand: per-token
                                      expert outputs, 2 * max_tokens * K * d fp32 */
  UNIF_MOE_FEATURES_DEFAULT = 3,   /* what unif_moe_create allocates */
  UNIF_MOE_FEATURES_ALL = 15
};
/* Expert GEMM kernels (all compute the same products; the fp32 sums into
 * the output differ only in order):
 * - EXPERT_TILE: rows grouped by expert, both projections of Eq. 16 in one
 *   kernel with h kept on chip, each (token, expert) added into the output
 *   once; bf16, d a multiple of 128 up to 384, H a multiple of 128, M a
 *   multiple of 64, a handle without UNIF_MOE_FEATURE_BACKWARD (otherwise
 *   as GROUPED).
 * - GROUPED: rows grouped by (expert, block) pair (Eq. 35's C_B pairs per
 *   token), an up and a down projection kernel with h in device memory;
 *   weight-stationary kernels where a group's weight slice fits in shared
 *   memory, else the streaming ones.
 * - STREAMING: as GROUPED, always the streaming kernels.
 * - AUTO: EXPERT_TILE where it applies, else GROUPED. */
enum {
  UNIF_MOE_GEMM_AUTO = 0,
  UNIF_MOE_GEMM_STREAMING = 1,
  UNIF_MOE_GEMM_GROUPED = 2,
  UNIF_MOE_GEMM_EXPERT_TILE = 3
};

typedef struct {
  unsigned int features; /* UNIF_MOE_FEATURE_* bits */
  int gemm_kernels;      /* UNIF_MOE_GEMM_AUTO, _STREAMING, _GROUPED, _EXPERT_TILE */
} unif_moe_options;

/* Fills *opts with the defaults of unif_moe_create: UNIF_MOE_FEATURES_DEFAULT
 * (norm-first sublayer and host-buffer forward), AUTO. */
UNIF_MOE_API void unif_moe_default_options(unif_moe_options* opts);

/* Creates a layer (Sec. III-A): d_model = d, d_ff = H, n_experts = K residual
 * experts (one shared expert is added), n_blocks = B, max_tokens = largest T
 * a forward will be given. th may be NULL (adaptive defaults).
 * Limits: 2 <= B <= 64, 1 <= K <= 64, H % B == 0, d % 8 == 0; for
 * UNIF_MOE_BF16 also d % 64 == 0 and M = H/B a multiple of 64.
 * Device workspace for max_tokens is allocated here, sized for the largest
 * possible C_B (Eq. 35) under th, with the buffers of the default features
 * (UNIF_MOE_FEATURES_DEFAULT); no later call allocates device memory.
 * Errors: ERR_ARG (out == NULL, bad values), ERR_SHAPE, ERR_CUDA (allocation). */
UNIF_MOE_API int unif_moe_create(unif_moe_t* out, int d_model, int d_ff, int n_experts, int n_blocks,
                    const unif_moe_thresholds* th, unif_moe_dtype dtype, int max_tokens);

/* unif_moe_create with options (NULL = the defaults above). A handle made
 * without a feature refuses the calls that need it with ERR_STATE, so no
 * later call allocates device memory either. Errors as unif_moe_create, and
 * ERR_ARG for unknown feature bits or GEMM kind. */
UNIF_MOE_API int unif_moe_create_ex(unif_moe_t* out, int d_model, int d_ff, int n_experts,
                                    int n_blocks, const unif_moe_thresholds* th,
                                    unif_moe_dtype dtype, int max_tokens,
                                    const unif_moe_options* opts);

/* Loads weights from device memory (copied into the handle; the caller may
 * free its buffers once `stream` has passed this call):
 *   w_router_dev [d][K+1]    column 0 = W_shr, columns 1..K = W_g (Eq. 17)
 *   w_up_dev     [K+1][H][d] expert 0 = shared; row h = key K_e[:, h] (Eq. 4)
 *   w_down_dev   [K+1][d][H] column h = value V_e[h, :] (Eq. 4)
 *   router_bias_dev [K+1] float or NULL: added to the router logits. The
 *                paper has no bias (Sec. II-A); NULL reproduces it.
 * Also forms the block prototypes mu_b (Eq. 20) from the shared keys, exactly
 * (fp64 sums) and rounded once to the layer dtype.
 * Errors: ERR_ARG (NULL weight), ERR_CUDA. */
UNIF_MOE_API int unif_moe_load_weights(unif_moe_t h, const void* w_router_dev, const void* w_up_dev,
                          const void* w_down_dev, const float* router_bias_dev, void* stream);

/* Upcycling (Sec. III: all experts start from the same dense FFN): loads the
 * dense FFN's projections into every expert, the shared one and the K
 * residual ones, then the router as unif_moe_load_weights does:
 *   w_router_dev    [d][K+1]  as in unif_moe_load_weights
 *   w_up_dense_dev  [H][d]    the dense FFN's keys, copied to every expert
 *   w_down_dense_dev [d][H]   the dense FFN's values, copied to every expert
 *   router_bias_dev [K+1] float or NULL
 * Layer dtype, device memory; copied, so the caller may free its buffers
 * once `stream` has passed this call. Errors: ERR_ARG (NULL weight), ERR_CUDA. */
UNIF_MOE_API int unif_moe_load_upcycled(unif_moe_t h, const void* w_router_dev,
                                        const void* w_up_dense_dev, const void* w_down_dense_dev,
                                        const float* router_bias_dev, void* stream);

/* One forward pass over T tokens (Eqs. 17-30):
 *   x_dev   [T][d] input tokens
 *   out_dev [T][d] output y (layer dtype); padding tokens give 0
 *   token_mask_dev [T] uint8 or NULL: 0 marks padding, which takes no routing
 *                decision, no expert work and outputs 0
 *   shared_counts_dev [T] int32 or NULL: receives b(x) (Eq. 19), 0 for padding
 *   residual_counts_dev [T] int32 or NULL: receives k(x) (Eq. 27), 0 for padding
 * T = 0 is a no-op. The decisions of the last forward stay in the handle for
 * unif_moe_get_routing / unif_moe_get_groups.
 * Errors: ERR_ARG, ERR_CAPACITY (T > max_tokens), ERR_STATE (no weights),
 * ERR_CUDA (launch failure). Kernel timeouts surface through sync_status. */
UNIF_MOE_API int unif_moe_forward(unif_moe_t h, const void* x_dev, void* out_dev, int T,
                     const uint8_t* token_mask_dev, int32_t* shared_counts_dev,
                     int32_t* residual_counts_dev, void* stream);

/* The layer as a Transformer sublayer, the way the paper's backbones hold
 * the converted FFN layers (Appendix A, Architecture details: DeiT-S normalises first, BERT after
 * the residual sum). With F the layer (Eqs. 16-30) and
 * LN(v) = gamma (v - mean(v)) / sqrt(var(v) + eps) + beta over each token's
 * d features (biased variance, fp32 statistics):
 *   norm_first != 0:  out = x + F(LN(x)), LN(x) kept in the layer dtype
 *   norm_first == 0:  out = LN(x + F(x))
 * ln_gamma_dev, ln_beta_dev [d] in the layer dtype (device); eps >= 0.
 * Padding tokens (mask 0) give 0. The routing decisions and counts are
 * those of F's input. x, out, counts, mask and errors as unif_moe_forward;
 * also ERR_ARG (NULL or not 16-byte aligned gamma or beta, bad eps),
 * ERR_SHAPE (d > 1024 or not a multiple of 8), ERR_STATE (norm_first on a
 * handle created without UNIF_MOE_FEATURE_NORM_FIRST; LN(x) goes to the
 * buffer allocated for it at create time). */
UNIF_MOE_API int unif_moe_sublayer_forward(unif_moe_t h, const void* x_dev, void* out_dev, int T,
                                           const uint8_t* token_mask_dev,
                                           int32_t* shared_counts_dev,
                                           int32_t* residual_counts_dev, const void* ln_gamma_dev,
                                           const void* ln_beta_dev, float eps, int norm_first,
                                           void* stream);

/* The same forward from host buffers: copies x_host (and token_mask_host if
 * not NULL) to the handle's device staging buffers, runs the forward, copies
 * the output to out_host and the counts to shared_counts_host /
 * residual_counts_host (each may be NULL), and synchronises `stream` before
 * returning. Host buffers should be pinned for asynchronous copies; output
 * buffers (out_host and the counts) in pinned host memory the device can
 * address are written by the kernels directly, with no copy back. The
 * staging buffers are allocated at create time (UNIF_MOE_FEATURE_HOST_IO;
 * ERR_STATE on a handle created without it). */
UNIF_MOE_API int unif_moe_forward_host(unif_moe_t h, const void* x_host, void* out_host, int T,
                          const uint8_t* token_mask_host, int32_t* shared_counts_host,
                          int32_t* residual_counts_host, void* stream);

/* Pipelined forwards from host buffers, for a stream of batches: enqueues
 * the forward of x_host and returns without waiting. Arguments and results
 * as unif_moe_forward_host (the same Eqs. 16-30; out_host [T][d] and the
 * counts receive this call's results), but the copies overlap other calls'
 * kernels: calls alternate between the handle's two staging slots, and a
 * call's input copy runs on a copy stream of the handle while the previous
 * call's kernels run on `stream`, its output copy on a second copy stream
 * while the next call's kernels run. A slot is refilled only after the
 * kernels two calls back have read it and their output has been copied out.
 * Ownership: the caller keeps x_host and token_mask_host unchanged, and does
 * not read out_host or the counts, until unif_moe_forward_host_wait has
 * returned; host buffers must be pinned (page-locked) for the copies to
 * overlap (pageable ones are still correct). Consecutive calls on one handle
 * pass the same `stream`; unif_moe_forward_host, unif_moe_get_routing and
 * the other calls that read the last forward's state come after
 * unif_moe_forward_host_wait. Errors: as unif_moe_forward_host (ERR_STATE
 * without UNIF_MOE_FEATURE_HOST_IO); a kernel timeout surfaces through
 * unif_moe_sync_status. Nothing is allocated. */
UNIF_MOE_API int unif_moe_forward_host_async(unif_moe_t h, const void* x_host, void* out_host,
                                             int T, const uint8_t* token_mask_host,
                                             int32_t* shared_counts_host,
                                             int32_t* residual_counts_host, void* stream);

/* Blocks until every forward enqueued by unif_moe_forward_host_async has
 * its output and counts in host memory. Errors: ERR_ARG (NULL handle),
 * ERR_STATE (handle without UNIF_MOE_FEATURE_HOST_IO), ERR_CUDA. */
UNIF_MOE_API int unif_moe_forward_host_wait(unif_moe_t h);

/* Backward pass of the last forward for training (Sec. III-E): given
 * dL/dy, the gradients of L with respect to x and to every parameter of
 * the layer, with the discrete decisions of that forward held fixed (the
 * rounding of Eq. 19, the TopK of Eq. 22 and the smallest prefix of Eq. 27
 * are piecewise constant): gradients flow through the pathway weights alpha
 * (Eq. 18) and s_j (Eq. 24) and through the experts (Eq. 16); the block
 * prototypes mu_b only rank blocks and have none. With lambda_div != 0 the
 * Gram regulariser L_div = ||W*^T W* - I_{K+1}||_F (Eq. diversity-loss) adds
 * lambda_div dL_div/dW* to the router gradient (the total loss of Eq. loss).
 *   x_dev  [T][d]   the input of that forward (layer dtype), unchanged
 *   dy_dev [T][d]   dL/dy (layer dtype)
 *   token_mask_dev  as given to that forward (padding gets dx = 0)
 * Outputs (fp32, device, overwritten):
 *   dx_dev        [T][d]        dL/dx
 *   dw_up_dev     [K+1][H][d]   dL/dw_up (the layout of unif_moe_load_weights)
 *   dw_down_dev   [K+1][d][H]   dL/dw_down
 *   dw_router_dev [d][K+1]      dL/dw_router (+ lambda_div dL_div/dW*)
 *   dbias_dev     [K+1] or NULL dL/d router bias
 *   l_div_dev     [1] or NULL   L_div
 * The weights are those last loaded. Needs a bf16 handle created with
 * UNIF_MOE_FEATURE_BACKWARD (ERR_STATE otherwise) and a forward of the same
 * T that ran in one pass (T <= unif_moe_pass_tokens; ERR_CAPACITY
 * otherwise); enqueued on `stream` after that forward, no sync. Pointers
 * 16-byte aligned. Errors: ERR_ARG, ERR_STATE, ERR_CAPACITY, ERR_CUDA. */
UNIF_MOE_API int unif_moe_backward(unif_moe_t h, const void* x_dev, const void* dy_dev, int T,
                                   const uint8_t* token_mask_dev, float* dx_dev,
                                   float* dw_up_dev, float* dw_down_dev, float* dw_router_dev,
                                   float* dbias_dev, float lambda_div, float* l_div_dev,
                                   void* stream);

/* Diagnostics of Sec. II-B, on the layer's K residual experts (experts 1..K
 * of the loaded weights) and their router columns: analysis tools, not part
 * of the forward. Handles created with UNIF_MOE_FEATURE_DIAGNOSTICS
 * (ERR_STATE otherwise), after a weight load. fp32 arithmetic.
 *
 * Value alignment (Eq. shared-set): for experts i, j (0-based among the
 * residual experts) and channel h, c_ijh = V_i[h,:] . V_j[h,:] /
 * (|V_i[h,:]| |V_j[h,:]|) (0 for a zero row), S_ij(delta) = {h : c_ijh >=
 * delta}; rho_dev [K][K] fp32 receives rho_ij = |S_ij| / H.
 * Errors: ERR_ARG (NULL rho, delta not finite), ERR_STATE, ERR_CUDA. */
UNIF_MOE_API int unif_moe_value_alignment(unif_moe_t h, float delta, float* rho_dev,
                                          void* stream);

/* Functional demand (Eqs. diagnostic-original .. functional-demand): for each
 * token of x_dev [T][d] (layer dtype), its top-2 pair (i, j) of
 * s = softmax(x W_g + bias) (the layer's router; ties to the lower index),
 * s~ = s / (s_i + s_j), y_orig = sum_{e in {i,j}} s~_e E_e(x), S_bar = the
 * same over the channels S_ij(delta), r = y_orig - S_bar, the residual order
 * q of x W_r (w_res_dev [d][K], layer dtype: the residual router, e.g. one
 * trained on the residual positions), R_m = E_{q_1..q_m} over the channels
 * outside S_ij, the ridge fit a* = (R_m R_m^T + gamma_m I)^{-1} R_m r with
 * gamma_m = 1e-6 tr(R_m R_m^T) / m (fp64; a = 0 when R_m = 0), and
 *   e_m = |a*^T R_m - r| / max(|y_orig|, 1e-12),  k_eps = min{m : e_m <= eps}
 * or the sentinel K + 1. Outputs (device): k_eps_dev [T] int32, err_dev
 * [T][K] fp32 (e_1..e_K) or NULL, pair_dev [T][2] int32 (i, j) or NULL.
 * Needs 2 <= K <= 32 (ERR_SHAPE) and T <= max_tokens (ERR_CAPACITY).
 * Errors also ERR_ARG, ERR_STATE, ERR_CUDA. */
UNIF_MOE_API int unif_moe_functional_demand(unif_moe_t h, const void* x_dev, int T,
                                            const void* w_res_dev, float delta, float eps,
                                            int32_t* k_eps_dev, float* err_dev,
                                            int32_t* pair_dev, void* stream);

/* Copies the decisions of the last forward (T tokens) to device buffers; any
 * pointer may be NULL:
 *   alpha_dev [T] float          shared demand alpha (Eq. 18)
 *   shared_mask_dev [T] uint64   bit b set = block b in I_shr (Eq. 22)
 *   expert_mask_dev [T] uint64   bit j set = residual expert j selected
 *   q_dev [T][K] int32           experts by decreasing affinity (Eq. 25)
 *   p_dev [T][K] float           their affinities p_1 >= ... >= p_K
 * Synchronises `stream`. Errors: ERR_ARG, ERR_STATE (no forward yet). */
UNIF_MOE_API int unif_moe_get_routing(unif_moe_t h, float* alpha_dev, uint64_t* shared_mask_dev,
                         uint64_t* expert_mask_dev, int32_t* q_dev, float* p_dev,
                         void* stream);

/* Copies the (expert, block) group table of the last forward to host memory
 * (of its last pass, tokens [T - n, T), when it ran in passes: see
 * unif_moe_pass_tokens).
 * Group g = e*B + b for e = 0 (shared expert) or e = 1+j (residual expert j),
 * G = (K+1)*B groups. counts_host [G] receives each group's row count; the
 * rows of group g are listed in increasing token order at
 * [offsets_host[g], offsets_host[g] + counts_host[g]) of row_token_host /
 * row_weight_host (weight = alpha for e = 0, p_i for e = 1+q_i). offsets_host
 * [G+1] (offsets_host[G] = total padded rows). Rows past a group's count up to
 * the next offset are padding (token -1). *n_rows receives offsets_host[G];
 * row buffers must hold max_rows entries, where unif_moe_max_rows() gives
 * the bound. Synchronises `stream`. */
UNIF_MOE_API int unif_moe_get_groups(unif_moe_t h, int32_t* counts_host, int32_t* offsets_host,
                        int32_t* row_token_host, float* row_weight_host, int64_t* n_rows,
                        void* stream);

/* Optional stage timing. events points to 6 cudaEvent_t handles created by
 * the caller (with timing enabled); each later forward records them on its
 * stream at the stage boundaries: [0] before the router, [1] after the
 * router (Eqs. 17-27), [2] after the permute (grouping of Eqs. 28-29),
 * [3] after the up-projection GEMM + GeLU, [4] after the down-projection
 * GEMM (Eq. 16), [5] after the combine (Eq. 30). A forward that runs in
 * passes records them around its last pass. NULL stops the recording.
 * The caller keeps the events alive while they are set. */
UNIF_MOE_API int unif_moe_set_stage_events(unif_moe_t h, void* const* events);

/* Upper bound on group-table rows (padded) of one pass of a forward. */
UNIF_MOE_API int64_t unif_moe_max_rows(unif_moe_t h);

/* Tokens per pass: bf16 layers run a forward of more tokens in consecutive
 * passes of this many tokens (the last one shorter), each pass the whole
 * layer (Eqs. 17-30) over its tokens, so that the fp32 output accumulator
 * of one pass (pass_tokens * d * 4 bytes, at most 128 MiB) stays resident
 * in L2. Results do not depend on it. max_tokens when a forward always runs
 * in one pass; -1 for a NULL handle. */
UNIF_MOE_API int unif_moe_pass_tokens(unif_moe_t h);

/* Number of kernels one pass of unif_moe_forward launches (a forward of
 * T > 0 tokens runs ceil(T / unif_moe_pass_tokens) passes): 4 for bf16
 * layers whose router also groups the pairs (router, up projection, down
 * projection, combine), 5 when a streaming GEMM reads a tile list, else 6
 * (router, group scan, group scatter, up, down, combine). -1 for a NULL
 * handle. */
UNIF_MOE_API int unif_moe_kernels_per_forward(unif_moe_t h);

/* Waits for `stream`, then reads and clears the handle's device status word.
 * Returns UNIF_MOE_OK, UNIF_MOE_ERR_TIMEOUT if a kernel abandoned a bounded
 * wait since the last call, or UNIF_MOE_ERR_CUDA. */
UNIF_MOE_API int unif_moe_sync_status(unif_moe_t h, void* stream);

/* Diagnostic: launches one kernel that waits, with its bounded wait, on a
 * barrier nothing ever completes, giving up after about `timeout_us`
 * microseconds (capped at 1 s) and recording ERR_TIMEOUT in the status word
 * exactly as the GEMM kernels would. Used to test the timeout path without
 * hanging the GPU. */
UNIF_MOE_API int unif_moe_selftest_timeout(unif_moe_t h, int timeout_us, void* stream);

/* Groups (expert, block) pairs by pair, like the grouping step inside
 * unif_moe_forward, but allocates nothing and needs no handle. It is for
 * callers that cannot call cudaMalloc: inference engines that plan all device
 * memory up front and give plugins no allocator once set up, and
 * latency-critical paths that cannot pay cudaMalloc's implicit device
 * synchronisation. The paper has no counterpart; this is a deployment aid.
 * Inputs (device, one entry per token, as unif_moe_get_routing returns them
 * plus the per-expert affinities):
 *   shared_mask_dev [T] uint64, expert_mask_dev [T] uint64, alpha_dev [T]
 *   float, affinity_dev [T][K] float (s_j by expert index j).
 * Outputs (device, caller-allocated): counts_dev [G], offsets_dev [G+1],
 *   n_tiles_dev [1], tile_group_dev and tile_row0_dev [row_capacity/128],
 *   row_token_dev and row_weight_dev [row_capacity]; G = (K+1)*B, layout as
 *   in unif_moe_get_groups (groups padded to 128 rows, padding token -1).
 * row_capacity must be at least T*K*B + G*127 (else ERR_CAPACITY).
 * Scratch: a 1 MiB array inside the library (device memory every GPU that
 * loads the library keeps until exit) holds the per-chunk counts, so
 * (K+1)*B*ceil(T/256) must not exceed 262144 (else ERR_CAPACITY). The first
 * call on each device looks up that array's device address; make that first
 * call before any stream capture. Calls that overlap on the GPU share the
 * array and race: order them on one stream. Enqueued on `stream`, no sync. */
UNIF_MOE_API int unif_moe_group_noalloc(int T, int n_experts, int n_blocks,
                                        const uint64_t* shared_mask_dev,
                                        const uint64_t* expert_mask_dev, const float* alpha_dev,
                                        const float* affinity_dev, int32_t* counts_dev,
                                        int32_t* offsets_dev, int32_t* n_tiles_dev,
                                        int32_t* tile_group_dev, int32_t* tile_row0_dev,
                                        int32_t* row_token_dev, float* row_weight_dev,
                                        int64_t row_capacity, void* stream);

/* Frees the handle and its device memory (synchronises the device first).
 * NULL is ignored. */
UNIF_MOE_API void unif_moe_destroy(unif_moe_t h);

/* Message of the last error on the calling thread ("" if none). */
UNIF_MOE_API const char* unif_moe_last_error(void);

#ifdef __cplusplus
}
#endif

#endif /* UNIF_MOE_H */
