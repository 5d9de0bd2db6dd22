// Internal launch interfaces of libprunepath (not part of the C ABI).
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

#include <algorithm>

#include "prunepath.h"

namespace pp {

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
    float* logit_ws;       // [T][E] scratch
    float* h_ws;           // [|U|][T][64] scratch
    unsigned* status;
    unsigned* bar;
    uint64_t timeout_ns;
    int T, d, E;
    int act, gate, rule;
    float p;
    int do_route, do_ffn;
    int R6, NS4, ded6, slots6, uch;
    uint32_t off_x, off_gw, off_mask, off_ulist, off_red, off_red6, off_ring6, off_ring4;
};

struct DecodePlanIn {
    int dtype, d, E, TS, grid;
    bool gated;
    size_t smem_limit;
};

struct DecodePlan {
    int R6, RPL, NS4, ded6, slots6, uch, threads;
    size_t smem;
    uint32_t off_x, off_gw, off_mask, off_ulist, off_red, off_red6, off_ring6, off_ring4;
};

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
cudaError_t wait_timeout_launch(unsigned* flag, unsigned* status, long long timeout_ns,
                                cudaStream_t st);

inline int sel_slots_for(int E) { return E <= 32 ? 1 : E <= 64 ? 2 : E <= 128 ? 4 : 8; }

}  // namespace pp
