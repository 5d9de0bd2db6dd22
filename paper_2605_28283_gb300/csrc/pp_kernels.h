// Internal launch interfaces of libprunepath (not part of the C ABI).
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

#include <algorithm>

#include <cuda_bf16.h>

#include "prunepath.h"

namespace pp {

// ---------------------------------------------------------------- rules
// Whether `rule` is one of the pp_rule values.
inline bool rule_known(int rule) { return rule >= PP_SEL_MIN_PREFIX && rule <= PP_SEL_LTE; }

// The rule parameter p (not NaN) in the form the selection kernels take:
// the mass budget for MIN_PREFIX / PAPER, the count k in [1, E] for TOPK,
// and for LTE the smallest fp32 logit g with sigmoid(g) > p (-inf for
// p <= 0: every logit; +inf for p >= 1: none).
float rule_kernel_param(int rule, float p, int E);

// ---------------------------------------------------------------- decode
struct DecodeArgs {
    CUtensorMap tmap_down;  // W_down [d][d_ff], box {64, R6}; must stay first (64-byte aligned)
    const void* x;
    const void* Wr;
    const void* Wg;
    const void* Wu;
    void* y;
    int32_t* sel_ids;      // route: outputs (CTA 0) or NULL; ffn-only: inputs
    int32_t* sel_counts;
    float* sel_gates;
    float* sel_logits;     // route: optional output
    unsigned long long* tlog;  // [T][E] tagged logits
    unsigned long long* th;    // [|U|][T][64] tagged gate/up activations
    unsigned* epochs;          // [grid] launch count per CTA (Control.epoch)
    unsigned* status;
    uint64_t timeout_ns;
    int T, d, E;
    int act, gate, rule;
    float p;
    int do_route, do_ffn;
    int R6, NS4, ded6, slots6, hch;
    uint32_t off_x, off_gw, off_mask, off_ulist, off_red, off_red6, off_ring6, off_ring4;
    // chained step: x = RMSNorm(x_prev + y_prev) * gamma computed in the
    // prologue (a.x is then x_prev); y_prev and gamma staged in the phase-4
    // ring at off_chain (free until phase 4), x written to x_out by CTA 0
    int chain;
    uint32_t off_chain;
    const void* y_prev;
    const void* gamma;
    void* x_out;
    float eps;
    // timeline instantiation only: [grid][kDecodeStamps] global-timer stamps
    unsigned long long* tline;
};

// Phase boundaries recorded by the decode kernel's timeline instantiation,
// per CTA (0 where a CTA skips the phase).
enum DecodeStamp {
    kStEntry = 0,    // first instruction
    kStReleased,     // the preceding grid on the stream has completed
    kStX,            // x (and the launch tag) in shared memory
    kStRouter,       // this CTA's router logits published
    kStSelected,     // every token's selection made (all logits received)
    kStUnion,        // union U of the activated experts formed
    kStIssued4,      // first gate/up row loads issued
    kStPhase4,       // this CTA's gate/up activations published
    kStFirstH,       // warp 0's first activations of phase 6 received
    kStPhase6,       // warp 0's down-projection products done
    kStEnd,          // y written (or the CTA's last phase done)
    kStLogits,       // cumulative-mass cut: every logit of token 0 received (warp 0)
    kStCut,          // cumulative-mass cut: warp 0's part of the count done
    kStCand,         // one-warp cut: candidates of token 0 formed (warp 0)
    kStLanded4,      // warp 0's first gate/up rows landed in shared memory
    kDecodeStamps = 16
};
// SM clock assumed by the timeline stamps between global-timer readings
// (the maximum clock of this GPU, which it runs at under this load)
constexpr long long kStampMHz = 2070;

struct DecodePlanIn {
    int dtype, d, E, TS, grid;
    bool gated;
    size_t smem_limit;
    bool chain = false;  // room for the chained step's y_prev and gamma
};

struct DecodePlan {
    int R6, RPL, NS4, ded6, slots6, hch, threads;
    size_t smem;
    uint32_t off_x, off_gw, off_mask, off_ulist, off_red, off_red6, off_ring6, off_ring4;
    uint32_t off_chain;  // within the phase-4 ring: y_prev [TS][d] then gamma [d]
};

// Part of the per-block shared-memory limit left to the decode kernel's
// static shared memory (selection scratch and counters, 4 KB once padded to
// the 1 KB alignment of the dynamic area).
constexpr size_t kDecodeStaticSmemReserve = 6144;

bool decode_plan(const DecodePlanIn& in, DecodePlan* out);
cudaError_t decode_launch(const DecodeArgs& a, const DecodePlan& p, int dtype, int TS, int grid,
                          cudaStream_t st);
int decode_max_ts(int dtype);

// --------------------------------------------------------- route / select
cudaError_t router_launch(int dtype, const void* x, int T, int d, const void* Wr, int E,
                          float* logits, cudaStream_t st);
cudaError_t select_launch(const float* logits, int T, int E, float p, int rule, int gate,
                          int32_t* ids, int32_t* counts, float* gates, unsigned* status,
                          cudaStream_t st);
cudaError_t stats_launch(const int32_t* counts, int T, int E, uint64_t* acc, cudaStream_t st);
// x[t] = RMSNorm(x_prev[t] + y_prev[t]) * gamma (y_prev, gamma nullable), one CTA per token
cudaError_t rmsnorm_residual_launch(int dtype, const void* x_prev, const void* y_prev, const void* gamma,
                                    float eps, int T, int d, void* x, cudaStream_t st);
int router_stats_blocks(int T);  // parts [blocks][E + 2] floats of router_stats_launch
cudaError_t router_stats_launch(const float* logits, int T, int E, float eps, float* part, double* out,
                                unsigned* status, cudaStream_t st);
cudaError_t wait_timeout_launch(unsigned* flag, unsigned* status, long long timeout_ns,
                                cudaStream_t st);

// ------------------------------------------------- tensor-core grouped path
struct GroupedPlan {
    int nk;          // 64-wide K chunks of d
    int kpb;         // router K chunks per split
    int nsplit;      // router K splits
    int max_items;   // upper bound on 128-row work items
    long long nnz_max;  // upper bound on (token, expert) assignments
    long long ycap;     // rows of the bf16 assignment-output buffer
};

struct GroupedArgs {
    GroupedPlan plan;
    const void* x;
    const void* Wr;
    const void* Wg;
    const void* Wu;
    const void* Wd;
    void* y;
    int T, d, E, act, gate, rule;
    float p;
    int32_t* ids;
    int32_t* counts;
    float* gates;
    float* logits_out;  // optional final logits
    float* part;        // [nsplit][T][E] router partials
    uint32_t* bits;     // [T][8]
    float* gexp;        // [T][E] gate weight per (token, expert)
    int* invpos;        // [T][E] permuted row of (token, expert)
    int* wcnt;          // [T/256][8][E] per-warp exclusive counts
    int* blkcnt;        // [T/256][E]
    int* blkbase;       // [T/256][E]
    int* offsets;       // [E + 1]
    void* items;        // [max_items] work items
    int* n_items;
    int* perm_token;    // [nnz_max]
    float* perm_gate;   // [nnz_max]
    __nv_bfloat16* H;   // [nnz_max + 128][64]
    __nv_bfloat16* Y;   // [ycap][d] assignment outputs
    float* yacc;        // [T][d] overflow accumulator, zero at rest
    int* overflow;      // set when any assignment went to yacc
    unsigned* status;
    uint64_t timeout_ns;
};

GroupedPlan grouped_plan(int T, int d, int E, int sms);
cudaError_t grouped_route(const GroupedArgs& a, cudaStream_t st);
cudaError_t grouped_ffn(const GroupedArgs& a, int sms, cudaStream_t st);

// ------------------------------------------------ MoEfication (Sec. 2.2)
// Balanced k-means over the neurons' input weights (host, offline); shapes
// and init already validated.  Returns PP_OK or PP_ERR_HOST.
pp_status moefy_cluster_host(int dtype, const void* Wg, const void* Wu, int dff, int d, int E, const int32_t* init,
                             int max_iter, int32_t* labels, int32_t* perm, int* iters, double* objective);
// perm check + row gather (W_gate, W_up) + column gather (W_down); Wg NULL for non-gated FFNs
cudaError_t moefy_permute_launch(int dtype, const int32_t* perm, const void* Wg, const void* Wu, const void* Wd,
                                 void* Wg_out, void* Wu_out, void* Wd_out, int d, int dff, int sms, unsigned* status,
                                 cudaStream_t st);

// cuTensorMapEncodeTiled through the runtime's driver entry point (nullptr if unavailable)
typedef CUresult (*TensorMapEncodeFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                      const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                      CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);
TensorMapEncodeFn tensor_map_encoder();

inline int sel_slots_for(int E) { return E <= 32 ? 1 : E <= 64 ? 2 : E <= 128 ? 4 : 8; }

}  // namespace pp
