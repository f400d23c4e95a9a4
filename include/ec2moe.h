/*
 * ec2moe.h - C ABI of libec2moe.so, the GB300 (sm_103a) MoE-layer forward of
 * EC^2MoE (arXiv 2508.06024).
 *
 * The layer computes Eq. 1, y = sum_i G(x)_i E_i(x), with the gate G of the
 * hardware-aware lightweight group gate network (Eq. 4 local candidate set,
 * Eq. 5 per-group softmax gates, Eq. 6 global group gate, Eq. 7 fusion), Top-k
 * routing (Top-1 in the paper's evaluation), and the low-rank encoder/decoder
 * of the end-cloud pipeline (Z = U^T X V at the end, X_hat = U_hat Z V_hat^T in
 * the cloud) at the split between gate/routing and the experts.
 *
 * Conventions shared by every entry point:
 *  - Device pointers are CUDA device addresses owned by the caller; the library
 *    never allocates, frees or keeps them.  Host pointers are marked "host".
 *  - Matrices are row-major and dense.  Weights are stored [out, in], i.e. the
 *    reduction axis is contiguous.  Every device pointer handed to a bf16
 *    tensor-core GEMM must be 16-byte aligned and every row a multiple of 16
 *    bytes (d, d_ff, r multiples of 8 for bf16); violations return
 *    EC2MOE_ERR_MISALIGNED before any launch.
 *  - Storage type: desc->dtype selects bf16 (EC2MOE_BF16) or fp32 (EC2MOE_F32)
 *    for activations, expert weights and codec weights.  Gate weights and
 *    biases are always fp32.  bf16 GEMMs accumulate in fp32.
 *  - All work is enqueued on `stream` (a cudaStream_t; NULL = legacy default
 *    stream).  No call synchronises except ec2moe_last_device_error.
 *  - Arguments are validated on the host before any launch; a failed check
 *    returns its status and enqueues nothing.  Kernels never trap: waits inside
 *    the tensor-core kernels are bounded and report through a device error
 *    word that ec2moe_last_device_error reads.
 *  - Calls are thread-safe with respect to each other as long as they do not
 *    share output buffers.
 */
#ifndef EC2MOE_H
#define EC2MOE_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct CUstream_st* ec2moe_stream_t; /* == cudaStream_t */

typedef enum ec2moe_status {
  EC2MOE_OK = 0,
  EC2MOE_ERR_INVALID_ARG = 1,      /* NULL pointer, non-positive size, E % n_groups != 0, ... */
  EC2MOE_ERR_ALL_MASKED = 2,       /* the local candidate set of Eq. 4 is empty */
  EC2MOE_ERR_TOO_FEW_EXPERTS = 3,  /* k > number of allowed experts */
  EC2MOE_ERR_UNSUPPORTED = 4,      /* a size beyond the limits below */
  EC2MOE_ERR_CUDA = 5,             /* a CUDA runtime call failed */
  EC2MOE_ERR_TIMEOUT = 6,          /* a bounded device wait gave up (see ec2moe_last_device_error) */
  EC2MOE_ERR_WORKSPACE = 7,        /* workspace NULL or smaller than ec2moe_workspace_size */
  EC2MOE_ERR_MISALIGNED = 8        /* pointer or row pitch not 16-byte aligned */
} ec2moe_status;

typedef enum ec2moe_dtype { EC2MOE_F32 = 0, EC2MOE_BF16 = 1 } ec2moe_dtype;

/* Expert FFN activation: GELU(u) = u Phi(u) (exact erf form), or SwiGLU
 * h = SiLU(W1 x) * (W3 x). */
typedef enum ec2moe_act { EC2MOE_GELU = 0, EC2MOE_SWIGLU = 1 } ec2moe_act;

#define EC2MOE_MAX_EXPERTS 128  /* E */
#define EC2MOE_MAX_GROUPS 16    /* K, n_groups */
#define EC2MOE_MAX_TOPK 8       /* k */
#define EC2MOE_MAX_SHARED 4     /* n_shared */

/* Shape of one MoE layer call.
 *  T            tokens (rows of X), >= 0 (T = 0 is a no-op)
 *  d            d_model
 *  E            routed experts (M of Eq. 5)
 *  d_ff         hidden width of each routed expert
 *  k            experts per token (Top-k)
 *  n_groups     K of Eq. 5-7; experts form K contiguous groups of E/K (group j
 *               owns experts [j*E/K, (j+1)*E/K)).  K = 1 is the plain softmax gate.
 *  act          ec2moe_act
 *  dtype        ec2moe_dtype
 *  r            codec rank; 0 = no codec (experts see X itself)
 *  n_shared     always-on shared experts (weight 1, not masked, not counted)
 *  d_ff_shared  hidden width of each shared expert
 *  renorm_topk  0: the combine weight is g_i itself (Eq. 1 with G = g);
 *               1: g_i divided by the sum of g over the token's top-k
 *  top_groups   0: every group takes part (Eq. 5-7).  G >= 1: top-group
 *               pruning, the group gate evaluated hierarchically -- per token
 *               only the G live groups (groups with an allowed expert) with
 *               the largest p_group of Eq. 6 keep their experts (ties to the
 *               lower group index, decided on the fp32 global logits), and
 *               p_group is renormalised over them, so the weights of Eq. 7
 *               still sum to 1 over the candidates.  G at or above the number
 *               of live groups (or K = 1) prunes nothing.  k above the allowed
 *               experts of the G live groups with the fewest returns
 *               EC2MOE_ERR_TOO_FEW_EXPERTS; G < 0 EC2MOE_ERR_INVALID_ARG. */
typedef struct ec2moe_layer_desc {
  int32_t T, d, E, d_ff, k, n_groups;
  int32_t act, dtype;
  int32_t r;
  int32_t n_shared, d_ff_shared;
  int32_t renorm_topk;
  int32_t top_groups;
} ec2moe_layer_desc;

/* Weights of one layer (device pointers, NULL where absent).
 *  W_local  fp32 [E, d]  the group gates W_k of Eq. 5 stacked in group order
 *  b_local  fp32 [E]     the b_k of Eq. 5 stacked likewise
 *  W_global fp32 [K, d]  Eq. 6 (NULL iff K == 1)
 *  b_global fp32 [K]     Eq. 6 (NULL iff K == 1)
 *  W1, W3   [E, d_ff, d] up projections (W3 only for SwiGLU)
 *  W2       [E, d, d_ff] down projection
 *  W1s, W3s [n_shared, d_ff_shared, d]; W2s [n_shared, d, d_ff_shared]
 *  V_enc    [r, d]       encoder: Z = X V_enc^T (V of the codec, U = I on tokens)
 *  V_dec    [d, r]       decoder: X_hat = Z V_dec^T (V_hat, U_hat = I) */
typedef struct ec2moe_layer_weights {
  const float* W_local;
  const float* b_local;
  const float* W_global;
  const float* b_global;
  const void* W1;
  const void* W3;
  const void* W2;
  const void* W1s;
  const void* W3s;
  const void* W2s;
  const void* V_enc;
  const void* V_dec;
} ec2moe_layer_weights;

/* Bytes of device workspace ec2moe_layer_forward needs for `desc` (0 on an
 * invalid desc).  The workspace holds the codec output Z, the decoded and
 * expert-ordered activations, the expert hidden activations, per-slot expert
 * outputs, the routing tables and the prepared gate rows; for decode-sized
 * bf16 calls (T <= 256) also the fp32 partial sums of the split-d_model gate,
 * the split-K encoder and the split-K down projection.  Its contents need no
 * initialisation and are not preserved between calls. */
size_t ec2moe_workspace_size(const ec2moe_layer_desc* desc);

/* Bytes of device workspace ec2moe_experts needs (hidden activations). */
size_t ec2moe_experts_workspace_size(const ec2moe_layer_desc* desc);

/* Bytes of device workspace ec2moe_route needs (per-block histograms). */
size_t ec2moe_route_workspace_size(const ec2moe_layer_desc* desc);

/* Steps 1-3a: local expert filter, group gate and Top-k.
 * Passage: Eq. 4 (the local candidate set E_local), Eq. 5 (per-group softmax
 * gates W_k x + b_k), Eq. 6 (global group gate W_global x + b_global), Eq. 7
 * (g_i = p_group^(k) p_local,i^(k)), and the Top-k selection of the gating
 * network that Eq. 1 sums over (Top-1 in the evaluation's parameter setup).
 *  X         [T, d] activations (dtype)
 *  mask      host uint8 [E]; 1 = expert in the local candidate set of Eq. 4.
 *            An all-zero mask returns EC2MOE_ERR_ALL_MASKED and fewer than k
 *            ones EC2MOE_ERR_TOO_FEW_EXPERTS.
 *  topk_idx  out int32 [T, k] expert ids, slot 0 = largest g, ties to the
 *            lower expert index
 *  topk_w    out fp32 [T, k] combine weights (g_i, or renormalised over the
 *            top-k when desc->renorm_topk)
 * Within a group the order is decided on the fp32 local logits; across groups
 * on the fp32 fused log-probability log p_group + log p_local. */
ec2moe_status ec2moe_gate(const ec2moe_layer_desc* desc, const void* X, const float* W_local,
                          const float* b_local, const float* W_global, const float* b_global,
                          const uint8_t* mask, int32_t* topk_idx, float* topk_w,
                          ec2moe_stream_t stream);

/* Step 3b: per-expert histogram, exclusive scan and stable permutation, plus
 * the optional gather of activation rows into expert order.
 * Passage: Eq. 1, whose sum runs only over the experts Top-k selected for each
 * token (Top-1 routing in the evaluation's parameter setup): the rows routed
 * to expert i are gathered so E_i runs once over all of them.
 *  topk_idx  int32 [T, k] (from ec2moe_gate)
 *  counts    out int32 [E]     tokens routed to each expert
 *  offsets   out int32 [E + 1] exclusive prefix sum of counts
 *  perm      out int32 [T * k] perm[p] = t * k + s for the p-th row in
 *            expert-major order; rows of one expert keep increasing (t, s)
 *  inv_perm  out int32 [T * k] or NULL: inv_perm[perm[p]] = p
 *  src, dst  NULL, or src [T, width] and dst [T * k, width] (dtype):
 *            dst[p] = src[perm[p] / k]
 *  workspace device scratch of ec2moe_route_workspace_size bytes
 * topk_idx is read on the device, so its ids cannot be checked before the
 * launch: an id outside [0, E) is skipped by the kernels (not counted, no perm
 * row, inv_perm = -1, no row gathered through it) and the next
 * ec2moe_last_device_error returns EC2MOE_ERR_INVALID_ARG; counts, offsets and
 * perm then describe the valid entries only. */
ec2moe_status ec2moe_route(const ec2moe_layer_desc* desc, const int32_t* topk_idx, int32_t* counts,
                           int32_t* offsets, int32_t* perm, int32_t* inv_perm, const void* src,
                           int32_t width, void* dst, void* workspace, size_t ws_bytes,
                           ec2moe_stream_t stream);

/* ec2moe_route without a workspace argument, for callers that cannot allocate
 * device memory: programs whose device memory is planned and reserved in full
 * before they start (a serving process that hands every byte to its own pool),
 * code in a latency-critical loop that must not hit cudaMalloc's implicit
 * device synchronisation, and bindings from languages that have no device
 * allocator of their own.  The paper has no counterpart; this is a library
 * convenience.
 *
 * Same arguments, results and errors as ec2moe_route except `workspace` and
 * `ws_bytes`.  The routing histograms live in a fixed 64 KiB device array
 * inside the library (EC2MOE_ROUTE_NOALLOC_MAX_CELLS int32 cells, one per
 * block of 1024 (token, slot) entries and expert), which every GPU that loads
 * the library holds until the process exits.  Sizes with
 * ceil(T * k / 1024) * E > EC2MOE_ROUTE_NOALLOC_MAX_CELLS (for E = 64: T * k >
 * 262144) return EC2MOE_ERR_UNSUPPORTED before any launch.  Nothing is
 * allocated or freed, by this call or by anything it calls.
 *
 * The first call on each device looks up the array's device address (with
 * that device current) and caches it, keyed on the device's current context;
 * make that first call before any stream capture.  After a cudaDeviceReset the
 * next call looks the address up again in the new context (so it, too, should
 * come before any capture), and the array's contents are gone.  All calls on a device share the array: every cell a call reads is
 * written earlier by the same call, but calls whose kernels overlap on the GPU
 * (different streams, or different host threads) race on it and must be
 * serialised by the caller. */
#define EC2MOE_ROUTE_NOALLOC_MAX_CELLS 16384
ec2moe_status ec2moe_route_noalloc(const ec2moe_layer_desc* desc, const int32_t* topk_idx, int32_t* counts,
                                   int32_t* offsets, int32_t* perm, int32_t* inv_perm, const void* src,
                                   int32_t width, void* dst, ec2moe_stream_t stream);

/* Steps 4-5a: routed expert FFNs on expert-ordered rows with the gate scale and
 * the unpermute fused into the down projection.
 * Passage: Eq. 1, each term G(x)_i E_i(x) with E_i a feed-forward expert
 * network (Preliminary, Mixture-of-Experts).
 *  X_perm    [T * k, d] rows in expert order (ec2moe_route's dst)
 *  offsets   int32 [E + 1] device (ec2moe_route)
 *  perm      int32 [T * k] device (ec2moe_route)
 *  topk_w    fp32 [T, k] (ec2moe_gate)
 *  slot_out  out [T * k, d]: slot_out[t * k + s] = topk_w[t, s] * E_e(x_t)
 *            for e = topk_idx[t, s]
 *  workspace ec2moe_experts_workspace_size bytes
 * offsets and perm are read on the device: a group whose range is not inside
 * [0, T * k] (or is decreasing) and a perm entry outside [0, T * k) are
 * skipped, with nothing written for them, and ec2moe_last_device_error then
 * reports EC2MOE_ERR_INVALID_ARG. */
ec2moe_status ec2moe_experts(const ec2moe_layer_desc* desc, const void* X_perm, const int32_t* offsets,
                             const void* W1, const void* W3, const void* W2, const float* topk_w,
                             const int32_t* perm, void* slot_out, void* workspace, size_t ws_bytes,
                             ec2moe_stream_t stream);

/* Always-on shared experts on every token: shared_out[s * T + t] = E_s(x_t).
 * Passage: Eq. 1's expert FFN E_i applied with weight 1 to every token; the
 * paper has no shared experts, the fine-grained layer shape adds them.
 *  X [T, d]; W1s/W3s/W2s as in ec2moe_layer_weights; shared_out out
 *  [n_shared * T, d]; workspace of ec2moe_experts_workspace_size bytes. */
ec2moe_status ec2moe_shared_experts(const ec2moe_layer_desc* desc, const void* X, const void* W1s,
                                    const void* W3s, const void* W2s, void* shared_out, void* workspace,
                                    size_t ws_bytes, ec2moe_stream_t stream);

/* Step 5b: y[t] = sum_s slot_out[t * k + s] + sum_j shared_out[j * T + t], in
 * that fixed order with an fp32 sum.  shared_out may be NULL.
 * Passage: Eq. 1, the sum over the selected experts of G(x)_i E_i(x). */
ec2moe_status ec2moe_combine(const ec2moe_layer_desc* desc, const void* slot_out, const void* shared_out,
                             void* Y, ec2moe_stream_t stream);

/* Step 6, end side: Z = X V_enc^T ([T, d] x [r, d]^T -> [T, r]).
 * Passage: the low-rank encoder of PO-ECC (Encoder-Decoder based on Low-Rank
 * Compression): Z = U^T X V, here with U = I on the token axis and
 * V = V_enc^T. */
ec2moe_status ec2moe_lr_encode(const ec2moe_layer_desc* desc, const void* X, const void* V_enc, void* Z,
                               ec2moe_stream_t stream);

/* Step 6, cloud side: X_hat = Z V_dec^T ([T, r] x [d, r]^T -> [T, d]).
 * Passage: the decoder of the same section, X_hat = U_hat Z V_hat^T, with
 * U_hat = I and V_hat = V_dec. */
ec2moe_status ec2moe_lr_decode(const ec2moe_layer_desc* desc, const void* Z, const void* V_dec,
                               void* X_hat, ec2moe_stream_t stream);

/* The fused layer: gate and routing on X, encode, decode into expert order,
 * routed and shared experts, combine.
 * Passage: Eq. 1 with the gate of Eq. 4-7 (HL-GGN) and the low-rank
 * encoder/decoder of PO-ECC at the end-cloud split between the gate and the
 * experts.
 *  Y         out [T, d] (dtype)
 *  topk_idx  out int32 [T, k]; topk_w out fp32 [T, k]; counts out int32 [E]
 *  Z         out [T, r] or NULL: the transmitted (encoded) activations
 *  workspace ec2moe_workspace_size(desc) bytes */
ec2moe_status ec2moe_layer_forward(const ec2moe_layer_desc* desc, const ec2moe_layer_weights* w,
                                   const void* X, const uint8_t* mask, void* Y, int32_t* topk_idx,
                                   float* topk_w, int32_t* counts, void* Z, void* workspace,
                                   size_t ws_bytes, ec2moe_stream_t stream);

/* Synchronises `stream`, then reads and clears the device error words of the
 * current device: EC2MOE_OK; EC2MOE_ERR_TIMEOUT when a bounded wait in a
 * tensor-core kernel gave up; EC2MOE_ERR_INVALID_ARG when a routing kernel met
 * (and skipped) an expert id outside [0, E) in a caller's topk_idx, or a
 * grouped expert GEMM met (and skipped) a group range in `offsets` outside
 * [0, T * k] or a destination in `perm` outside [0, T * k); EC2MOE_ERR_CUDA
 * when the stream reports an error.  A timeout takes precedence. */
ec2moe_status ec2moe_last_device_error(ec2moe_stream_t stream);

/* Budget, in SM clock cycles, of every bounded wait inside the tensor-core
 * kernels of later calls (process-wide; default 4e9, about two seconds).  A
 * wait that runs out makes its CTA stop, wait (with a fixed one-second
 * budget) for the copies and MMAs it started, free its tensor memory and
 * return; ec2moe_last_device_error then reports EC2MOE_ERR_TIMEOUT and the
 * context stays usable.  A budget of 0 makes every wait that is not already
 * satisfied give up at once, which is how failure handling is exercised
 * without a real fault.  Negative values return EC2MOE_ERR_INVALID_ARG. */
ec2moe_status ec2moe_set_wait_budget(int64_t cycles);
int64_t ec2moe_get_wait_budget(void);

/* ---------------------------------------------------------------------------
 * The end/cloud pipeline of the paper's pipeline optimisation (PO-ECC: the end
 * runs the gate and the low-rank encoder, the cloud the decoder and the
 * experts, overlapped across requests), on one GPU with two CUDA streams.
 *
 * Same result as ec2moe_layer_forward, computed in n_micro contiguous
 * micro-batches of ceil(T / n_micro) tokens: stream_end runs the gate, the
 * routing and the encoder Z = X V_enc^T of micro-batch i + 1 while
 * stream_cloud runs the decoder (rows straight into expert order), the
 * experts, the shared experts and the combine of micro-batch i.  The
 * micro-batch's Z and routing tables are handed from the end to the cloud
 * through a CUDA event; counts is the sum of the micro-batches' histograms.
 * Y, topk_idx, topk_w and Z (optional) receive every token's rows in token
 * order, as for ec2moe_layer_forward; the order of rows inside each expert
 * (not an output) follows the micro-batches.
 *
 * Streams: stream_cloud first waits for everything enqueued on stream_end
 * before the call, and at the end stream_end waits for stream_cloud, so the
 * call as a whole is ordered on stream_end (synchronise or capture on
 * stream_end; stream_cloud is forked and joined inside the call).  Passing the
 * same stream twice runs the micro-batches back to back.
 *
 * workspace: ec2moe_pipelined_workspace_size(desc, n_micro) bytes, 16-byte
 * aligned; one region per micro-batch, so calls that overlap on the GPU must
 * not share it.  1 <= n_micro <= EC2MOE_MAX_MICRO (else
 * EC2MOE_ERR_INVALID_ARG); micro-batches beyond T tokens are empty and
 * skipped.  Other errors as ec2moe_layer_forward. */
#define EC2MOE_MAX_MICRO 64
size_t ec2moe_pipelined_workspace_size(const ec2moe_layer_desc* desc, int32_t n_micro);
ec2moe_status ec2moe_layer_forward_pipelined(const ec2moe_layer_desc* desc, const ec2moe_layer_weights* w,
                                             const void* X, const uint8_t* mask, void* Y, int32_t* topk_idx,
                                             float* topk_w, int32_t* counts, void* Z, void* workspace,
                                             size_t ws_bytes, int32_t n_micro, ec2moe_stream_t stream_end,
                                             ec2moe_stream_t stream_cloud);

/* Number of kernels the last successful call on this host thread enqueued. */
int32_t ec2moe_last_launch_count(void);

/* Per-launch timing.  While enabled, every kernel the library enqueues is
 * bracketed by a pair of CUDA events recorded on its stream; records
 * accumulate until ec2moe_profile_reset.  Reading a record synchronises on its
 * stop event.  `name` receives a static string naming the launch
 * ("gate_prep", "gate_topk", "gate_decide", "route_count", "route_scatter", "gather_rows",
 * "lr_encode", "lr_reduce", "lr_decode", "lr_codec", "expert_up", "expert_down", "shared_up",
 * "shared_down", "combine", "sum_counts"); `ms` its device duration.  Profiling is off by default and
 * costs nothing when off. */
ec2moe_status ec2moe_profile_enable(int32_t enable);
/* Restricts profiling to one launch per call: with launch_index >= 0 only the
 * kernel that is the launch_index-th launch (0-based) of each later call is
 * bracketed, so its neighbours run without event records between them (which
 * would otherwise end the programmatic overlap of every launch with its
 * predecessor and add the records' own cost to every measured kernel);
 * -1 (the default) brackets every launch.  Values below -1 return
 * EC2MOE_ERR_INVALID_ARG. */
ec2moe_status ec2moe_profile_only(int32_t launch_index);
int32_t ec2moe_profile_count(void);
ec2moe_status ec2moe_profile_read(int32_t i, const char** name, float* ms);
void ec2moe_profile_reset(void);

/* ---------------------------------------------------------------------------
 * Route-aware heuristic pipeline scheduler (Eq. 9-11 of the paper's pipeline
 * optimisation).  Host code only: no device memory, no CUDA call, no stream.
 * Every pointer below is a host pointer.
 *
 * ec2moe_schedule places n tasks, task i with computational complexity
 * cost[i] = C(t_i) >= 0 and communication cost comm[i] = Comm(t_i) >= 0, on
 * the End (location[i] = EC2MOE_END) or the Cloud (EC2MOE_CLOUD):
 *   Eq. 10  P(t_i) = C(t_i) / (Comm(t_i) + eps)
 *   Eq. 11  End if Load_end + C(t_i) <= T_end and P(t_i) >= beta, else Cloud,
 * visiting the tasks in decreasing priority (ties to the lower index) and
 * adding C(t_i) to Load_end (starting at load_end) for each End task and to
 * Load_cloud (starting at load_cloud; reported only, Eq. 11 does not use it)
 * for each Cloud task.  order[j] receives the j-th visited task (may be NULL);
 * *load_end_out and *load_cloud_out the final loads (may be NULL).
 * Errors: EC2MOE_ERR_INVALID_ARG for n < 0, NULL cost/comm/location when
 * n > 0, a negative or NaN cost or comm, eps < 0 or NaN, or comm[i] + eps == 0
 * for some i.  T_end and beta may be +/-infinity. */
#define EC2MOE_END 0
#define EC2MOE_CLOUD 1
ec2moe_status ec2moe_schedule(int32_t n, const double* cost, const double* comm, double load_end,
                              double load_cloud, double T_end, double beta, double eps, int32_t* location,
                              int32_t* order, double* load_end_out, double* load_cloud_out);

/* Eq. 9, the heuristic's objective for a placement:
 *   sum_i alpha * ExecTime(t_i) + (1 - alpha) * Comm(t_i),
 * with ExecTime(t_i) = cost[i] / rate_end on the End and cost[i] / rate_cloud
 * on the Cloud, and Comm(t_i) paid by Cloud tasks only (a task run on the End
 * transmits nothing).  Sums in task order.  Errors: EC2MOE_ERR_INVALID_ARG for
 * n < 0, NULL arrays when n > 0, rates <= 0, a location other than
 * EC2MOE_END / EC2MOE_CLOUD, or NULL `objective`. */
ec2moe_status ec2moe_schedule_objective(int32_t n, const double* cost, const double* comm,
                                        const int32_t* location, double rate_end, double rate_cloud,
                                        double alpha, double* objective);

/* Route-aware tasks from a layer's routing histogram (counts, host copy of
 * the [E] output of ec2moe_route / ec2moe_layer_forward): one task per expert
 * with rows, in expert order.  expert_of_task[j] is the expert of task j,
 * cost[j] = 2 * rows * d * d_ff * (3 projections for SwiGLU, 2 for GELU) its
 * FFN flops, comm[j] = rows * (w_in + d) * bytes its transfer in bytes if it
 * runs in the Cloud (w_in = r encoded values per row, or d without a codec;
 * plus the d-wide output row; bytes = 2 for bf16, 4 for fp32).  All output
 * arrays hold desc->E entries; *n_tasks receives the task count.  Errors:
 * EC2MOE_ERR_INVALID_ARG for NULL pointers, an invalid desc, or a negative
 * count. */
ec2moe_status ec2moe_expert_tasks(const ec2moe_layer_desc* desc, const int32_t* counts, int32_t* expert_of_task,
                                  double* cost, double* comm, int32_t* n_tasks);

/* Human-readable name of a status code (static storage). */
const char* ec2moe_status_string(ec2moe_status status);

#ifdef __cplusplus
}
#endif

#endif /* EC2MOE_H */
