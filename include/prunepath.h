/*
 * prunepath.h -- C ABI of the GB300 (sm_103a) PrunePath sparse-FFN library.
 *
 * PrunePath (Sec. 3.1) routes each token x in R^d with a linear router
 *   g = W_r^T x                                   (Eq. routing_logits)
 *   p_j = exp(g_j) / sum_i exp(g_i)               (Eq. softmax_prob)
 * orders the experts by descending probability (pi), activates a prefix of
 * that order by cumulative probability mass     (Eq. tau_thresh_activate)
 * and evaluates only the activated expert slices of a MoEfied FFN
 *   y = sum_{e in A} sigmoid(g_e) * FFN_e(x)      (Eq. moe_output)
 * where FFN_e is the restriction of the gated FFN (Eq. ffn) to the e-th block
 * of d_e contiguous intermediate neurons        (Eq. moefication_decomp).
 *
 * ------------------------------------------------------------------------
 * Conventions shared by every entry point
 *  - Every tensor pointer is a DEVICE pointer owned by the caller, row-major,
 *    contiguous and 16-byte aligned.  The library never allocates, frees or
 *    keeps a tensor pointer beyond the call.  The one exception is the
 *    offline host routine pp_moefy_cluster, whose pointers are host pointers.
 *  - Weight layout ("expert neurons stored contiguously"):
 *      W_r    [E][d]      row j is the routing vector of expert j
 *                         (the paper's W_r in R^{d x E}, stored transposed)
 *      W_gate [d_ff][d]   row n holds neuron n's input weights; expert e is
 *      W_up   [d_ff][d]   the dense row block [e*d_e, (e+1)*d_e)
 *      W_down [d][d_ff]   expert e is the dense column block [e*d_e, (e+1)*d_e)
 *    x and y are [T][d].  Element type: pp_desc.dtype for x, y and all weights.
 *  - The selection (pp_selection) is [T][E] int32 ids in rank order (first
 *    counts[t] entries valid, the rest -1), counts [T] int32, gates [T][E]
 *    fp32 aligned with ids (sigmoid(g_e) for PP_GATE_SIGMOID, 1 for
 *    PP_GATE_NONE, 0 past counts[t]) and, optionally, logits [T][E] fp32 in
 *    expert order.
 *  - Every call is asynchronous on `stream` (a cudaStream_t passed as void*;
 *    NULL means the legacy default stream).  Argument errors are returned
 *    synchronously before anything is enqueued.  Errors found on the device
 *    (a bounded wait that timed out, a non-finite logit) are recorded in the
 *    workspace status word and read back by pp_get_device_status.
 *  - Workspace: caller-owned device memory of at least pp_workspace_size()
 *    bytes, 256-byte aligned, zeroed once by pp_workspace_init before its
 *    first use.  Calls that share a workspace must be ordered on one stream;
 *    calls on different workspaces are independent.  A workspace serves one
 *    device (it keeps per-SM launch counts of the fused decode kernel).
 *  - No C++ exception crosses this interface.
 *  - Supported shapes: d_expert == 64, d_ff == E * 64, 1 <= E <= 256,
 *    d a multiple of 8 (bf16) or 4 (fp32), 64 <= d <= 8192, T >= 0.
 *    Other shapes return PP_ERR_SHAPE.
 *  - p is the parameter of the cut rule (pp_desc.rule); NaN returns
 *    PP_ERR_INVALID_ARG under every rule.
 *      MIN_PREFIX, PAPER: the mass budget tau.  p >= 1 activates all E
 *        experts (the warm-up setting tau_warm = 1.05 of Sec. 3.2); p <= 0
 *        activates the top-1 expert only.
 *      TOPK: the expert count k = floor(p), at least 1 and at most E.
 *      LTE: the score threshold delta; p <= 0 activates all E experts and
 *        p >= 1 none (counts[t] = 0, y[t] = 0).
 */
#ifndef PRUNEPATH_H
#define PRUNEPATH_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum pp_status {
    PP_OK = 0,
    PP_ERR_INVALID_ARG = 1, /* NULL pointer, NaN p, unknown enum value            */
    PP_ERR_SHAPE = 2,       /* shape outside the supported set (see above)        */
    PP_ERR_DTYPE = 3,       /* unsupported dtype / activation combination         */
    PP_ERR_ALIGN = 4,       /* a pointer is not 16-byte aligned                   */
    PP_ERR_WORKSPACE = 5,   /* workspace NULL, misaligned or too small            */
    PP_ERR_CUDA = 6,        /* a CUDA runtime call failed (launch, attribute)     */
    PP_ERR_TIMEOUT = 7,     /* device: a bounded wait gave up (sticky)            */
    PP_ERR_CAPACITY = 8,    /* device: an internal buffer would overflow (sticky) */
    PP_ERR_NONFINITE = 9,   /* device: a router logit was NaN/Inf (sticky); the
                               token gets counts[t] = 0 and y[t] = 0              */
    PP_ERR_UNSUPPORTED = 10,/* no device of compute capability 10.3 is current    */
    PP_ERR_HOST = 11        /* host memory or threads could not be obtained (the
                               offline host routine pp_moefy_cluster)             */
} pp_status;

typedef enum pp_dtype { PP_F32 = 0, PP_BF16 = 1 } pp_dtype;

/* FFN variant.  SWIGLU is Eq. (ffn) with phi = SiLU and needs W_gate; RELU
   and GELU_TANH are the non-gated forms h = phi(x W_up) (Sec. 2.1 notes the
   analysis covers any FFN separable along d_ff) and take W_gate = NULL. */
typedef enum pp_act { PP_ACT_RELU = 0, PP_ACT_GELU_TANH = 1, PP_ACT_SWIGLU = 2 } pp_act;

/* Output weighting.  SIGMOID is Eq. (moe_output); NONE weights every
   selected expert by 1, the plain decomposition of Eq. (moefication_decomp). */
typedef enum pp_gate { PP_GATE_SIGMOID = 0, PP_GATE_NONE = 1 } pp_gate;

/* Activation rule on the router logits g.  Every rule lists the activated
   experts in the descending order pi (ties by lower expert index).
   MIN_PREFIX: the shortest prefix of pi whose mass reaches p (keeps the rank
   that crosses p).  PAPER: Eq. (tau_thresh_activate) literally, rank 1 plus
   every rank with S_i < p.  Whenever S_E >= p, |PAPER| =
   max(1, |MIN_PREFIX| - 1).
   TOPK: the first k = floor(p) experts of pi, the fixed expert budget of the
   top-k reconstruction analysis (Sec. 4.3).
   LTE: every expert with sigmoid(g_e) > p, each expert thresholded on its
   own (Eq. lte_hard_set, the rule PrunePath is compared with in Sec. 2.3);
   LTE's own aggregation (Eq. lte_hard_output) is PP_GATE_NONE.  The device
   takes the same decision on the fp32 logit: g_e >= the smallest fp32 value
   above ln(p / (1 - p)), a bound the host computes in double precision. */
typedef enum pp_rule { PP_SEL_MIN_PREFIX = 0, PP_SEL_PAPER = 1, PP_SEL_TOPK = 2, PP_SEL_LTE = 3 } pp_rule;

typedef struct pp_desc {
    int d_model;   /* d                                   */
    int d_ff;      /* intermediate width, == n_experts*64 */
    int n_experts; /* E                                   */
    int d_expert;  /* d_e, must be 64                     */
    int dtype;     /* pp_dtype                            */
    int act;       /* pp_act                              */
    int gate;      /* pp_gate                             */
    int rule;      /* pp_rule                             */
} pp_desc;

typedef struct pp_selection {
    int32_t *ids;    /* [T][E] device, rank order, -1 padded          */
    int32_t *counts; /* [T]    device                                 */
    float *gates;    /* [T][E] device, aligned with ids               */
    float *logits;   /* [T][E] device, expert order; may be NULL      */
} pp_selection;

/* Bytes of workspace needed for calls with up to T tokens. */
size_t pp_workspace_size(const pp_desc *desc, int T);

/* Zero the whole workspace (status word, launch counts, accumulators) on
   `stream`.  Call once after allocating a workspace, and again to clear a
   sticky device error. */
pp_status pp_workspace_init(void *ws, size_t ws_bytes, void *stream);

/* Router and selection (Eq. routing_logits, softmax_prob,
   tau_thresh_activate).  x [T][d], W_r [E][d]; writes *out (out->logits may
   be NULL).  The softmax is max-shifted in fp32 with fp32 exponentials; the
   normaliser and the prefix masses are summed exactly (2^-31 fixed-point
   integers for up to 64 tokens per call, fp64 beyond), so the cut is decided
   by an exact comparison with p times the normaliser; the order is
   descending logit with ties broken by the lower expert index. */
pp_status pp_route(const pp_desc *desc, const void *x, int T, const void *W_r, float p,
                   const pp_selection *out, void *ws, size_t ws_bytes, void *stream);

/* Selection only, from given fp32 logits [T][E] (out->logits is ignored). */
pp_status pp_select(const pp_desc *desc, const float *logits, int T, float p,
                    const pp_selection *out, void *ws, size_t ws_bytes, void *stream);

/* Sparse FFN over a given selection (Eq. moe_output): for each token t,
   y[t] = sum_{r < counts[t]} gates[t][r] * FFN_{ids[t][r]}(x[t]).
   Reads sel->ids, sel->counts, sel->gates.  W_gate is NULL unless act is
   PP_ACT_SWIGLU.  Accumulation is fp32; y has the dtype of x. */
pp_status pp_sparse_ffn(const pp_desc *desc, const void *x, int T, const void *W_gate,
                        const void *W_up, const void *W_down, const pp_selection *sel, void *y,
                        void *ws, size_t ws_bytes, void *stream);

/* pp_route followed by pp_sparse_ffn, fused where the token count allows.
   sel_out may be NULL (the selection then stays in the workspace). */
pp_status pp_layer(const pp_desc *desc, const void *x, int T, const void *W_r, const void *W_gate,
                   const void *W_up, const void *W_down, float p, const pp_selection *sel_out,
                   void *y, void *ws, size_t ws_bytes, void *stream);

/* One layer of a chained decode step: the layer input is formed from the
   previous layer's input and output,
     x = RMSNorm(x_prev + y_prev) * gamma,   RMSNorm(v) = v / sqrt(mean(v^2) + eps)
   per token (the post-norm residual connection x_{l+1} = RMSNorm(x_l + y_l)
   that stacks the layers of the decode setting of Sec. 4.5), written to x,
   and then y = pp_layer(x).  x_prev, y_prev, x, y are [T][d]; gamma is [d];
   y_prev may be NULL (no residual term: the first layer) and gamma NULL
   (unit weights).  The sum and the mean square are fp32; x is stored in the
   desc dtype and the layer reads exactly that x.  For up to 4 bf16 / 8 fp32
   tokens the fused decode kernel forms x in its prologue (one launch);
   otherwise one more kernel runs first.  x and y must not overlap x_prev,
   y_prev or each other (PP_ERR_INVALID_ARG); eps >= 0. */
pp_status pp_layer_chained(const pp_desc *desc, const void *x_prev, const void *y_prev, const void *gamma,
                           float eps, int T, const void *W_r, const void *W_gate, const void *W_up,
                           const void *W_down, float p, const pp_selection *sel_out, void *x, void *y, void *ws,
                           size_t ws_bytes, void *stream);

/* pp_layer for callers that cannot allocate device memory where they run a
   layer -- a runtime that has given every byte to its own pool, a loop that
   must not block on an allocation's implicit synchronisation, a plug-in host
   that exposes no allocator.  The paper has no counterpart: this entry point
   exists only for those callers.
   Same computation and arguments as pp_layer, for T <= 4 tokens and without a
   workspace.  Like pp_layer, it runs the tokens in slices when one fused
   launch cannot hold them all (fp32 rows of a wide model).  Its scratch (status word, per-CTA launch counts, router
   logits and gate/up activations: 533,760 bytes) is one static
   device array that every GPU loading this library keeps until the process
   exits; no call allocates or frees.
   - T > 4 (like any shape pp_layer rejects) returns PP_ERR_SHAPE.
   - The first call on a device, made with that device current, looks up the
     array's address there; make that first call before any stream capture.
   - Every call reuses the same array and first clears its status word;
     calls that overlap on the GPU (other streams, other host threads) race
     on it, so the caller must serialise them.
   - status_out (optional, device uint32) receives the call's device-side
     status (a pp_status code) when the call has run on `stream`. */
pp_status pp_layer_noalloc(const pp_desc *desc, const void *x, int T, const void *W_r,
                           const void *W_gate, const void *W_up, const void *W_down, float p,
                           const pp_selection *sel_out, void *y, uint32_t *status_out, void *stream);

/* FFN-sparsity statistics (Sec. 4.1, s_FFN): adds sum_t counts[t] to
   acc[0] and a histogram of counts (0..E) to acc[1..E+1].  acc is
   [E+2] uint64 on the device, accumulated across calls (one per layer), so
   s_FFN = 1 - acc[0] / (N * L * E). */
pp_status pp_sparsity_stats(const int32_t *counts, int T, int n_experts, uint64_t *acc,
                            void *stream);

/* Router statistics of a batch of B = T tokens (forward values of the router
   terms of the training objective, reported as routing diagnostics):
     out[0] = L_ent  = -(1/B) sum_t sum_j p_tj log(p_tj + eps)  (Sec. 3.2, Eq. entropy_loss)
     out[1] = L_bal  = E sum_j ((1/B) sum_t p_tj)^2             (Sec. 3.2, Eq. load_balance_loss)
     out[2] = L_gate = (1/(B E)) sum_t sum_j sigmoid(g_tj)       (Sec. 4.2.3, gate-magnitude term)
   with p_tj the softmax of Eq. (softmax_prob).  logits [T][E] fp32 device
   (e.g. the logits pp_route writes); out: 3 doubles, device, 8-byte aligned.
   The softmax is max-shifted in fp32; the sums are fp32 in a fixed order,
   pairwise across blocks of 64 tokens, combined in fp64 (deterministic).  T >= 1 (else PP_ERR_SHAPE); eps NaN is
   PP_ERR_INVALID_ARG.  Uses the workspace of pp_workspace_size(desc, T).  A
   non-finite logit records PP_ERR_NONFINITE and makes out[0] NaN. */
pp_status pp_router_stats(const pp_desc *desc, const float *logits, int T, float eps, double *out, void *ws,
                          size_t ws_bytes, void *stream);

/* MoEfication preprocessing, clustering (Sec. 2.2): group the d_ff
   intermediate neurons of a dense FFN into E experts of d_e = 64 neurons by
   balanced k-means over their input weights, and return the permutation Pi
   that makes every expert a contiguous block (pp_moefy_permute applies it).
   An OFFLINE HOST routine, run once per model before serving: W_gate, W_up,
   init, perm, labels, iters and objective are HOST pointers; it runs on the
   calling thread and a pool of host threads and touches no GPU.
   - Features: neuron n's input weights -- row n of W_gate followed by row n
     of W_up for PP_ACT_SWIGLU (W_gate required), row n of W_up otherwise
     (W_gate ignored); W_gate, W_up are [d_ff][d] in desc->dtype, widened
     exactly.
   - Balanced k-means (the constrained k-means of Bradley, Bennett and
     Demiriz, 2000, with every cluster holding exactly 64 neurons): the
     centroids start at the features of neurons init[0..E) (distinct, in
     [0, d_ff); the random choice is the caller's); each iteration assigns
     the neurons to clusters with the least total squared Euclidean distance
     under the equal-size constraint (solved exactly, fp64), then moves every
     centroid to the mean of its members; it stops when an assignment repeats
     the previous one, or after max_iter (>= 1) assignments.
   - Outputs: perm [d_ff] int32 (new position j holds old neuron perm[j];
     cluster e fills positions [64e, 64e + 64) in ascending old index);
     labels [d_ff] int32, the cluster of each old neuron (may be NULL);
     *iters = assignments made and *objective = the last assignment's sum of
     squared distances (either may be NULL).
   - Host memory: about d_ff * (f * 4 + E * 8) bytes, f = d or 2d.
   Errors: PP_ERR_INVALID_ARG (NULL input or perm, bad init, max_iter < 1),
   PP_ERR_SHAPE / PP_ERR_DTYPE as for every call, PP_ERR_HOST. */
pp_status pp_moefy_cluster(const pp_desc *desc, const void *W_gate, const void *W_up, const int32_t *init,
                           int max_iter, int32_t *perm, int32_t *labels, int *iters, double *objective);

/* MoEfication preprocessing, repacking (Eq. permuted_weights:
   W~_gate = W_gate Pi, W~_up = W_up Pi, W~_down = Pi^T W_down).  With the
   neurons stored as rows of W_gate / W_up and columns of W_down:
     W_gate_out[j][:] = W_gate[perm[j]][:],  W_up_out[j][:] = W_up[perm[j]][:],
     W_down_out[:][j] = W_down[:][perm[j]]
   so that expert e of the MoEfied FFN is the block of new neurons
   [64e, 64e + 64) that every other call of this library reads.  Device
   pointers: perm [d_ff] int32; weights in desc->dtype; W_gate / W_gate_out
   are used only for PP_ACT_SWIGLU (required then).  No output may overlap an
   input or another output (PP_ERR_INVALID_ARG).  Device-side check: an
   entry of perm outside [0, d_ff), or repeated, records PP_ERR_INVALID_ARG
   in the workspace status (pp_get_device_status); rows and columns for
   out-of-range entries are written as zeros.  Workspace:
   pp_workspace_size(desc, 0) bytes, initialised. */
pp_status pp_moefy_permute(const pp_desc *desc, const int32_t *perm, const void *W_gate, const void *W_up,
                           const void *W_down, void *W_gate_out, void *W_up_out, void *W_down_out, void *ws,
                           size_t ws_bytes, void *stream);

/* Synchronise `stream` and return the sticky device status of `ws`. */
pp_status pp_get_device_status(void *ws, void *stream);

/* Diagnostic: pp_layer for one bf16 token (T = 1) through the timeline
   instantiation of the fused decode kernel, which computes the same y and
   also records the GPU global timer (ns) at the phase boundaries of every
   CTA: stamps[CTA * 16 + i] for i = first instruction, preceding grid
   complete, x loaded, router logits published, selection made, union formed,
   gate/up loads issued, gate/up activations published, first activations of
   the down projection received, down products done, y written (0 where a CTA
   skips a phase: the caller zeroes stamps first, so that consecutive layers
   need nothing between their launches).  stamps: device uint64, at least
   256 * 16 entries (stamps_bytes).  Errors as pp_layer; a dtype
   other than bf16 is PP_ERR_DTYPE. */
pp_status pp_debug_decode_timeline(const pp_desc *desc, const void *x, const void *W_r, const void *W_gate,
                                   const void *W_up, const void *W_down, float p, void *y, void *ws,
                                   size_t ws_bytes, uint64_t *stamps, size_t stamps_bytes, void *stream);

/* Test hook for failure detection: enqueue one kernel that waits on a
   workspace flag nothing sets, with a limit of timeout_ns nanoseconds; it
   then records PP_ERR_TIMEOUT in the workspace status and returns.  No GPU
   fault, trap or hang is involved. */
pp_status pp_debug_wait_timeout(void *ws, size_t ws_bytes, long long timeout_ns, void *stream);

/* Human-readable name of a status code (static string). */
const char *pp_status_string(pp_status s);

/* Library version, "major.minor.patch". */
const char *pp_version(void);

#ifdef __cplusplus
}
#endif

#endif /* PRUNEPATH_H */
