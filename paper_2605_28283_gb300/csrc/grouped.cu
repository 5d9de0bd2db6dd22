// Tensor-core (tcgen05) path for many tokens: batched decode and prefill.
//
//   router GEMM   logits = X W_r^T (Eq. routing_logits), split over K; the
//                 selection kernel sums the K-split partials in fixed order
//   dispatch      per-token expert bitmasks -> per-expert counts -> offsets
//                 and 128-row work items -> a stable permutation (tokens in
//                 ascending order within each expert) with each assignment's
//                 gate weight
//   grouped G/U   per work item (expert e, <= 128 of its tokens):
//                 D[128 x (64|128)] = X_gathered * [W_gate_e ; W_up_e]^T on
//                 tcgen05 (TMA gather4 for the token rows), then
//                 h = act(gate, up) * gate weight (Eq. ffn, Eq. moe_output),
//                 stored bf16 in permuted order
//   grouped down  per work item and 256-wide slice j of d:
//                 D[128 x 256] = H_item * W_down[j, e-block]^T (K = 64); each
//                 row (one token-expert assignment) is stored bf16 in the
//                 permuted order
//   combine       y[t] = sum over t's experts, in ascending expert order, of
//                 its assignment rows (fp32 accumulation, deterministic)
//   Assignments past the row buffer's capacity (only near-dense selections)
//   are added into an fp32 accumulator with vector reductions instead; the
//   combine step reads and re-zeroes it.
//
// Every GEMM kernel: warp 0 = TMA producer, warp 1 = TMEM owner and UMMA
// issuer (one thread), warps 2..5 = epilogue (TMEM lanes 32*(warp%4)..).
// All waits are bounded (PP_ERR_TIMEOUT).
#include "pp_common.cuh"
#include "pp_kernels.h"
#include "pp_select.cuh"
#include "pp_tc.cuh"

namespace pp {

constexpr int kTcThreads = 192;
constexpr int kTileBytesA = 128 * 128;  // 128 rows x 64 bf16

struct WorkItem {
    int e, a0, cnt, pad;
};

// ====================================================================== router
// Grid (m-tiles, splits).  CTA (m, s): D[128 tokens x NE] over K chunks
// [s*kpb, min((s+1)*kpb, nk)); partial logits to part[s][t][e].
template <int NE>
__global__ void __launch_bounds__(kTcThreads, 1)
    router_gemm_kernel(const __grid_constant__ CUtensorMap map_x, const __grid_constant__ CUtensorMap map_wr,
                       int T, int E, int nk, int kpb, float* part, unsigned* status, uint64_t lim) {
    pdl_wait();  // the previous kernel on the stream has completed (programmatic dependent launch)
    pdl_launch_dependents();
    constexpr int kStages = 4;
    constexpr int kTileB = NE * 128;
    constexpr int kStage = kTileBytesA + kTileB;
    extern __shared__ __align__(1024) unsigned char smem_raw[];
    unsigned char* smem = reinterpret_cast<unsigned char*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);
    __shared__ uint64_t full[kStages], empty[kStages], tfull;
    __shared__ uint32_t taddr_s;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int m0 = blockIdx.x * 128, split = blockIdx.y;
    const int k0 = split * kpb, k1 = min(nk, k0 + kpb);
    if (threadIdx.x == 0) {
        for (int i = 0; i < kStages; i++) {
            mbar_init(&full[i], 1);
            mbar_init(&empty[i], 1);
        }
        mbar_init(&tfull, 1);
        fence_mbar_init();
    }
    if (warp == 1) {
        tmem_alloc(&taddr_s, NE <= 128 ? 128 : 256);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = taddr_s;

    if (warp == 0 && lane == 0) {
        for (int kc = k0, it = 0; kc < k1; kc++, it++) {
            const int s = it % kStages;
            if (it >= kStages) mbar_wait(&empty[s], (uint32_t)((it / kStages) - 1) & 1u, status, lim);
            unsigned char* st = smem + (size_t)s * kStage;
            mbar_arrive_expect_tx(&full[s], kStage);
            tma_load_2d(st, &map_x, kc * 64, m0, &full[s]);
            tma_load_2d(st + kTileBytesA, &map_wr, kc * 64, 0, &full[s]);
        }
    } else if (warp == 1 && lane == 0) {
        constexpr uint32_t idesc = idesc_bf16_m128(NE);
        for (int kc = k0, it = 0; kc < k1; kc++, it++) {
            const int s = it % kStages;
            mbar_wait(&full[s], (uint32_t)(it / kStages) & 1u, status, lim);
            tc_fence_after();
            unsigned char* st = smem + (size_t)s * kStage;
            umma_k64(tmem, st, st + kTileBytesA, idesc, it > 0);
            umma_commit(&empty[s]);
        }
        umma_commit(&tfull);
    } else if (warp >= 2) {
        // lane = row 32 q + lane of the tile; 32 x 32 blocks are transposed
        // through shared memory (the pipeline stages are free once every MMA
        // has completed) so that each store writes 32 consecutive logits of
        // one row
        const int q = warp & 3;
        mbar_wait(&tfull, 0, status, lim);
        tc_fence_after();
        float* tr = reinterpret_cast<float*>(smem) + (size_t)(warp - 2) * 32 * 33;
#pragma unroll 1
        for (int c = 0; c < NE; c += 32) {
            uint32_t r[32];
            tmem_ld32(tmem + ((uint32_t)(32 * q) << 16) + (uint32_t)c, r);
            tmem_ld_wait();
#pragma unroll
            for (int i = 0; i < 32; i++) tr[lane * 33 + i] = k1 > k0 ? __uint_as_float(r[i]) : 0.0f;
            __syncwarp();
            for (int i = 0; i < 32; i++) {
                const int t = m0 + 32 * q + i;
                if (t < T && c + lane < E) part[((size_t)split * T + t) * E + c + lane] = tr[i * 33 + lane];
            }
            __syncwarp();
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 1) tmem_dealloc(tmem, NE <= 128 ? 128 : 256);
}

// ================================================================= selection
// Selection from K-split partial logits (summed in split order).  Up to
// kCtaSelectMaxTokens tokens take one CTA each (the counting selection);
// beyond, one warp per token (the warp sort).
constexpr int kCtaSelectMaxTokens = 256;

// Logit = sum over s of part[s * stride + off], added in split order; the
// loads go out 8 at a time instead of one dependent round trip each.
PP_DEVINL float sum_partials(const float* __restrict__ part, int nsplit, size_t stride, size_t off) {
    float v = 0.0f;
    int s = 0;
    for (; s + 8 <= nsplit; s += 8) {
        float q[8];
#pragma unroll
        for (int i = 0; i < 8; i++) q[i] = __ldg(part + (size_t)(s + i) * stride + off);
#pragma unroll
        for (int i = 0; i < 8; i++) v += q[i];
    }
    for (; s < nsplit; s++) v += __ldg(part + (size_t)s * stride + off);
    return v;
}

template <int S>
__global__ void __launch_bounds__(256) select_part_kernel(const float* __restrict__ part, int nsplit, int T, int E,
                                                          float p, int rule, int gate, int32_t* ids, int32_t* counts,
                                                          float* gates, float* logits_out, unsigned* status) {
    pdl_wait();  // the previous kernel on the stream has completed (programmatic dependent launch)
    pdl_launch_dependents();
    const int lane = threadIdx.x & 31;
    const int t = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
    if (t >= T) return;
    auto load = [&](int j) { return sum_partials(part, nsplit, (size_t)T * E, (size_t)t * E + j); };
    unsigned long long key[S];
    bool finite = true;
    const int k = warp_select<S>(load, E, p, rule, key, &finite);
    if (!finite && lane == 0) record_status(status, PP_ERR_NONFINITE);
#pragma unroll
    for (int s = 0; s < S; s++) {
        const int r = lane * S + s;
        if (r >= E) continue;
        const bool on = finite && r < k;
        ids[(size_t)t * E + r] = on ? key_index(key[s]) : -1;
        gates[(size_t)t * E + r] = on ? gate_of(gate, key[s]) : 0.0f;
    }
    if (lane == 0) counts[t] = k;
    if (logits_out)
        for (int j = lane; j < E; j += 32) logits_out[(size_t)t * E + j] = load(j);
}

__global__ void __launch_bounds__(256) select_part_cta_kernel(const float* __restrict__ part, int nsplit, int T,
                                                              int E, float p, int rule, int gate, int32_t* ids,
                                                              int32_t* counts, float* gates, float* logits_out,
                                                              unsigned* status) {
    pdl_wait();  // the previous kernel on the stream has completed (programmatic dependent launch)
    pdl_launch_dependents();
    __shared__ __align__(16) CtaSelScratch sc;
    const int t = blockIdx.x;
    auto load = [&](int j) { return sum_partials(part, nsplit, (size_t)T * E, (size_t)t * E + j); };
    bool on;
    int r;
    float g;
    const int k = cta_select_fn(load, E, p, rule, true, sc, status, &on, &r, &g);
    const int j = threadIdx.x;
    write_selection_row(ids + (size_t)t * E, gates + (size_t)t * E, j, E, k, on, r,
                        on ? (gate == PP_GATE_NONE ? 1.0f : sigmoidf_(g)) : 0.0f);
    if (j < E && logits_out) logits_out[(size_t)t * E + j] = g;
    if (j == 0) counts[t] = k;
}

// Cumulative-mass cut (MIN_PREFIX / PAPER with p < 1) of any number of
// tokens: one CTA per token runs the three-barrier cut of the fused decode
// kernel on the summed partial logits.
__global__ void __launch_bounds__(256) select_part_cut_kernel(const float* __restrict__ part, int nsplit, int T, int E,
                                                              float p, int rule, int gate, int32_t* ids,
                                                              int32_t* counts, float* gates, float* logits_out,
                                                              unsigned* status) {
    pdl_wait();  // the previous kernel on the stream has completed (programmatic dependent launch)
    pdl_launch_dependents();
    __shared__ __align__(16) CutShared sc;
    __shared__ __align__(16) WarpCand cand[256];
    const int t = blockIdx.x, j = threadIdx.x;
    const float g = j < E ? sum_partials(part, nsplit, (size_t)T * E, (size_t)t * E + j) : -INFINITY;
    int32_t* idr = ids + (size_t)t * E;
    float* gtr = gates + (size_t)t * E;
    const int k = cta_mass_cut(g, E, p, rule, sc, cand, status, [&](int r, int e, float ge) {
        idr[r] = e;
        gtr[r] = gate == PP_GATE_NONE ? 1.0f : sigmoidf_(ge);
    }, [] {});
    for (int r = k + j; r < E; r += 256) {
        idr[r] = -1;
        gtr[r] = 0.0f;
    }
    if (j < E && logits_out) logits_out[(size_t)t * E + j] = g;
    if (j == 0) counts[t] = k;
}

// ================================================================== dispatch
// bits[t][w]: bit (e % 32) of word e / 32 set when token t activated e;
// gexp[t][e]: the gate weight of that assignment (gates of a repeated id
// add up), 0 where e is not activated.  Invalid ids and counts are recorded
// and skipped.
__global__ void __launch_bounds__(256) dispatch_bits_kernel(const int32_t* __restrict__ ids,
                                                            const int32_t* __restrict__ counts,
                                                            const float* __restrict__ gates, int T, int E,
                                                            uint32_t* bits, float* gexp, unsigned* status) {
    pdl_wait();  // the previous kernel on the stream has completed (programmatic dependent launch)
    pdl_launch_dependents();
    // one warp per token: coalesced row writes
    const int lane = threadIdx.x & 31;
    const int t = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
    if (t >= T) return;
    float* grow = gexp + (size_t)t * E;
    for (int e = lane; e < E; e += 32) grow[e] = 0.0f;
    int k = counts[t];
    if (k < 0 || k > E) {
        if (lane == 0) record_status(status, PP_ERR_INVALID_ARG);
        k = k < 0 ? 0 : E;
    }
    __syncwarp();
    uint32_t w[8] = {0, 0, 0, 0, 0, 0, 0, 0};
    // entries in rank order, one lane each; repeated ids add their gates in
    // rank order (the lanes of a round take turns on a repeated id)
    for (int r0 = 0; r0 < k; r0 += 32) {
        const int r = r0 + lane;
        int e = r < k ? ids[(size_t)t * E + r] : -1;
        if (r < k && (e < 0 || e >= E)) {
            record_status(status, PP_ERR_INVALID_ARG);
            e = -1;
        }
        const float gv = e >= 0 ? gates[(size_t)t * E + r] : 0.0f;
        if (e >= 0) w[e >> 5] |= 1u << (e & 31);
        for (int l = 0; l < 32; l++) {
            const int el = __shfl_sync(kFull, e, l);
            const float gl = __shfl_sync(kFull, gv, l);
            if (el >= 0 && lane == (el & 31)) grow[el] += gl;
            __syncwarp();
        }
    }
#pragma unroll
    for (int i = 0; i < 8; i++) {
        uint32_t v = w[i];
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) v |= __shfl_xor_sync(kFull, v, o);
        if (lane == i) bits[(size_t)t * 8 + i] = v;
    }
}

// Token block b (256 tokens, one per thread): per-warp counts of every
// expert via ballots; block totals blkcnt[b][e].
constexpr int kDispBlock = 256;

__global__ void __launch_bounds__(kDispBlock) dispatch_count_kernel(const uint32_t* __restrict__ bits, int T, int E,
                                                                    int* wcnt, int* blkcnt) {
    pdl_wait();  // the previous kernel on the stream has completed (programmatic dependent launch)
    pdl_launch_dependents();
    const int b = blockIdx.x, lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int t = b * kDispBlock + threadIdx.x;
    uint32_t w[8];
#pragma unroll
    for (int i = 0; i < 8; i++) w[i] = t < T ? bits[(size_t)t * 8 + i] : 0u;
    __shared__ int sc[8][kMaxExperts];
    for (int e = 0; e < E; e++) {
        const unsigned bal = __ballot_sync(kFull, (w[e >> 5] >> (e & 31)) & 1u);
        if (lane == 0) sc[warp][e] = __popc(bal);
    }
    __syncthreads();
    for (int e = threadIdx.x; e < E; e += kDispBlock) {
        int s = 0;
        for (int v = 0; v < 8; v++) {
            wcnt[((size_t)b * 8 + v) * E + e] = s;  // exclusive prefix over the block's warps
            s += sc[v][e];
        }
        blkcnt[(size_t)b * E + e] = s;
    }
}

// One block, thread e: hist, offsets (exclusive scan over experts), the
// per-token-block bases and the expert's 128-row work items; clears the
// overflow flag of the down projection.
__global__ void __launch_bounds__(kMaxExperts) dispatch_scan_kernel(const int* __restrict__ blkcnt, int nblk, int E,
                                                                    int* offsets, int* blkbase, WorkItem* items,
                                                                    int* n_items, int* overflow) {
    pdl_wait();  // the previous kernel on the stream has completed (programmatic dependent launch)
    pdl_launch_dependents();
    const int e = threadIdx.x;
    if (e == 0) *overflow = 0;  // the down projection's overflow flag starts clear
    __shared__ int sh[kMaxExperts], si[kMaxExperts];
    int h = 0;
    if (e < E)
        for (int b = 0; b < nblk; b++) h += blkcnt[(size_t)b * E + e];
    sh[e] = e < E ? h : 0;
    si[e] = e < E ? (h + 127) / 128 : 0;
    __syncthreads();
    if (e == 0) {  // exclusive scans of counts and item counts (E <= 256)
        int a = 0, n = 0;
        for (int i = 0; i < E; i++) {
            const int c = sh[i], m = si[i];
            sh[i] = a;
            si[i] = n;
            a += c;
            n += m;
        }
        offsets[E] = a;
        *n_items = n;
    }
    __syncthreads();
    if (e >= E) return;
    const int off = sh[e];
    offsets[e] = off;
    int base = off;
    for (int b = 0; b < nblk; b++) {
        blkbase[(size_t)b * E + e] = base;
        base += blkcnt[(size_t)b * E + e];
    }
    int n = si[e];
    for (int m = 0; m < h; m += 128) items[n++] = WorkItem{e, off + m, min(128, h - m), 0};
}

// Token block b again: each token writes itself (and its gate weight) at
// base + (earlier warps) + (earlier lanes) for every activated expert, so
// tokens stay in ascending order within each expert; invpos[t][e] records
// where (t, e) landed.
__global__ void __launch_bounds__(kDispBlock) dispatch_scatter_kernel(const uint32_t* __restrict__ bits,
                                                                      const float* __restrict__ gexp, int T, int E,
                                                                      const int* __restrict__ wcnt,
                                                                      const int* __restrict__ blkbase,
                                                                      int* perm_token, float* perm_gate,
                                                                      int* invpos) {
    pdl_wait();  // the previous kernel on the stream has completed (programmatic dependent launch)
    pdl_launch_dependents();
    const int b = blockIdx.x, lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int t = b * kDispBlock + threadIdx.x;
    const bool live = t < T;
    // experts [e0, e1) of this block (blockIdx.y splits the expert loop)
    const int e0 = blockIdx.y * E / gridDim.y, e1 = (blockIdx.y + 1) * E / gridDim.y;
    // this block's bases, per warp: blkbase[b][e] + wcnt[b][warp][e]
    __shared__ int base_s[8][kMaxExperts];
    for (int i = threadIdx.x; i < 8 * (e1 - e0); i += kDispBlock) {
        const int v = i / (e1 - e0), e = e0 + i - v * (e1 - e0);
        base_s[v][e] = blkbase[(size_t)b * E + e] + wcnt[((size_t)b * 8 + v) * E + e];
    }
    __syncthreads();
    uint32_t w[8];
#pragma unroll
    for (int i = 0; i < 8; i++) w[i] = live ? bits[(size_t)t * 8 + i] : 0u;
    const unsigned lt = (1u << lane) - 1u;
    for (int e = e0; e < e1; e++) {
        const bool on = (w[e >> 5] >> (e & 31)) & 1u;
        const unsigned bal = __ballot_sync(kFull, on);
        if (on) {
            const int pos = base_s[warp][e] + __popc(bal & lt);
            perm_token[pos] = t;
            perm_gate[pos] = gexp[(size_t)t * E + e];
            invpos[(size_t)t * E + e] = pos;
        }
    }
}

// All of the dispatch for T <= 256 tokens in one CTA of 1024 threads (small
// batches are latency-bound: four kernels with a serial loop over the
// experts cost more than their work).  Shared memory holds, per expert, the
// 256-bit mask of the tokens that activated it; an assignment (t, e) lands
// at offsets[e] + (tokens below t in e's mask), so tokens stay in ascending
// order within each expert, as in the multi-block path; work items hold at
// most item_rows rows.  Writes the same
// outputs as that path (bits, offsets, work items, perm_token, perm_gate,
// invpos) and clears the overflow flag of the down projection.  Gates of a
// repeated id add up (with three or more copies the order of the additions
// is not fixed).
constexpr int kSmallDispatchMaxT = 256;

__global__ void __launch_bounds__(1024) dispatch_small_kernel(const int32_t* __restrict__ ids,
                                                              const int32_t* __restrict__ counts,
                                                              const float* __restrict__ gates, int T, int E,
                                                              uint32_t* bits, int* offsets, WorkItem* items,
                                                              int* n_items, int* perm_token, float* perm_gate,
                                                              int* invpos, int* overflow, int item_rows,
                                                              unsigned* status) {
    pdl_wait();  // the previous kernel on the stream has completed (programmatic dependent launch)
    pdl_launch_dependents();
    __shared__ uint32_t mask[kMaxExperts][8];              // tokens of expert e
    __shared__ uint32_t dup[kSmallDispatchMaxT][8];        // entry (t, r) repeats an earlier id of token t
    __shared__ int off_s[kMaxExperts + 1], item_s[kMaxExperts + 1];
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    for (int i = tid; i < kMaxExperts * 8; i += blockDim.x) {
        (&mask[0][0])[i] = 0u;
        (&dup[0][0])[i] = 0u;
    }
    if (tid == 0) *overflow = 0;
    __syncthreads();
    // warp w takes tokens w + 32 i, lane r their entries r, r + 32, ...; the
    // count and entry r = lane of each of the warp's tokens are read once, all
    // loads independent (the three passes below reuse them)
    constexpr int kTokPerWarp = kSmallDispatchMaxT / 32;
    int ck[kTokPerWarp], ce[kTokPerWarp];
    float cg[kTokPerWarp];
#pragma unroll
    for (int i = 0; i < kTokPerWarp; i++) {
        const int t = warp + 32 * i;
        ck[i] = 0;
        ce[i] = -1;
        cg[i] = 0.0f;
        if (t < T) {
            ck[i] = counts[t];
            if (lane < E) {
                ce[i] = ids[(size_t)t * E + lane];
                cg[i] = gates[(size_t)t * E + lane];
            }
        }
    }
    // token masks
#pragma unroll
    for (int i = 0; i < kTokPerWarp; i++) {
        const int t = warp + 32 * i;
        if (t >= T) break;
        int k = ck[i];
        if (k < 0 || k > E) {
            if (lane == 0) record_status(status, PP_ERR_INVALID_ARG);
            k = k < 0 ? 0 : E;
        }
        ck[i] = k;
        for (int r = lane; r < k; r += 32) {
            const int e = r == lane ? ce[i] : ids[(size_t)t * E + r];
            if (e < 0 || e >= E) {
                record_status(status, PP_ERR_INVALID_ARG);
                continue;
            }
            const uint32_t bit = 1u << (t & 31);
            if (atomicOr(&mask[e][t >> 5], bit) & bit) atomicOr(&dup[t][r >> 5], 1u << (r & 31));
        }
    }
    __syncthreads();
    // per-expert counts -> offsets and work items (warp 0 scans, 8 experts per lane)
    if (warp == 0) {
        int c[8], m[8], cs = 0, ms = 0;
#pragma unroll
        for (int q = 0; q < 8; q++) {
            const int e = lane * 8 + q;
            int n = 0;
            if (e < E)
#pragma unroll
                for (int w = 0; w < 8; w++) n += __popc(mask[e][w]);
            c[q] = n;
            m[q] = (n + item_rows - 1) / item_rows;
            cs += n;
            ms += m[q];
        }
        int ci = cs, mi = ms;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int cv = __shfl_up_sync(kFull, ci, o), mv = __shfl_up_sync(kFull, mi, o);
            if (lane >= o) {
                ci += cv;
                mi += mv;
            }
        }
        int ce = ci - cs, me = mi - ms;
#pragma unroll
        for (int q = 0; q < 8; q++) {
            off_s[lane * 8 + q] = ce;
            item_s[lane * 8 + q] = me;
            ce += c[q];
            me += m[q];
        }
        if (lane == 31) {
            off_s[kMaxExperts] = ci;
            item_s[kMaxExperts] = mi;
        }
    }
    __syncthreads();
    if (tid < E) {
        const int e = tid, o = off_s[e], n = off_s[e + 1] - o;
        offsets[e] = o;
        int it = item_s[e];
        for (int a0 = 0; a0 < n; a0 += item_rows) items[it++] = WorkItem{e, o + a0, min(item_rows, n - a0), 0};
    }
    if (tid == 0) {
        offsets[E] = off_s[kMaxExperts];
        *n_items = item_s[kMaxExperts];
    }
    // bits[t][w]: bit i of word w = token t activated expert 32 w + i
    for (int q = tid; q < T * 8; q += blockDim.x) {
        const int t = q >> 3, w = q & 7;
        uint32_t v = 0;
        for (int i = 0; i < 32 && 32 * w + i < E; i++) v |= ((mask[32 * w + i][t >> 5] >> (t & 31)) & 1u) << i;
        bits[(size_t)t * 8 + w] = v;
    }
    // scatter: the first entry of each (t, e) writes its slot, repeats add
    // their gate afterwards
    for (int pass = 0; pass < 2; pass++) {
#pragma unroll
        for (int i = 0; i < kTokPerWarp; i++) {
            const int t = warp + 32 * i;
            if (t >= T) break;
            const int k = ck[i];
            for (int r = lane; r < k; r += 32) {
                const int e = r == lane ? ce[i] : ids[(size_t)t * E + r];
                if (e < 0 || e >= E) continue;
                const bool rep = (dup[t][r >> 5] >> (r & 31)) & 1u;
                if (rep != (pass == 1)) continue;
                int pos = off_s[e] + __popc(mask[e][t >> 5] & ((1u << (t & 31)) - 1u));
                for (int w = 0; w < (t >> 5); w++) pos += __popc(mask[e][w]);
                const float gv = r == lane ? cg[i] : gates[(size_t)t * E + r];
                if (pass == 0) {
                    perm_token[pos] = t;
                    perm_gate[pos] = gv;
                    invpos[(size_t)t * E + e] = pos;
                } else {
                    atomicAdd(&perm_gate[pos], gv);
                }
            }
        }
        __syncthreads();
    }
}

// =============================================================== grouped G/U
// Persistent over work items.  NB = 128 (SwiGLU: gate rows then up rows) or
// 64 (non-gated: up rows).  Two TMEM accumulators let the epilogue of one
// item overlap the MMAs of the next.
//
// Warp roles: warp 0 streams the expert's weight tiles with 2-D TMA, warp 1
// issues the MMAs, warps 2-5 run the epilogue, and warps 6-9 gather the
// item's token rows: thread r copies row r of the A tile (128 bytes per
// K chunk) with eight 16-byte cp.async into the 128-byte-swizzled layout the
// TMA would write.  (A TMA gather4 moves 512 bytes per instruction and its
// rate, about 14 GB/s per SM, bounded this kernel; cp.async keeps the L2
// streaming.)  A gather thread keeps kGatherLag stages of copies in flight;
// once a stage's copies are complete it fences them into the async proxy
// and arrives on the stage's full barrier (129 arrivals: the weight TMA's
// expect-tx arrival and the 128 gather threads).
constexpr int kGuThreads = 320;
constexpr int kGatherLag = 3;

template <int NB>
__global__ void __launch_bounds__(kGuThreads, 1)
    gu_gemm_kernel(const __nv_bfloat16* __restrict__ x, int d, const __grid_constant__ CUtensorMap map_wg,
                   const __grid_constant__ CUtensorMap map_wu, const WorkItem* __restrict__ items,
                   const int* __restrict__ n_items_p, const int* __restrict__ perm_token,
                   const float* __restrict__ perm_gate, int nk, int act, __nv_bfloat16* H, unsigned* status,
                   uint64_t lim) {
    pdl_wait();  // the previous kernel on the stream has completed (programmatic dependent launch)
    pdl_launch_dependents();
    constexpr int kStages = NB == 128 ? 6 : 8;
    static_assert(kGatherLag < kStages, "a gather thread must release a stage before it waits for it again");
    constexpr int kTileB = NB * 128;
    constexpr int kStage = kTileBytesA + kTileB;
    constexpr uint32_t kCols = 2 * NB;  // two accumulators
    extern __shared__ __align__(1024) unsigned char smem_raw[];
    unsigned char* smem = reinterpret_cast<unsigned char*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);
    __shared__ uint64_t full[kStages], empty[kStages], tfull[2], tempty[2];
    __shared__ uint32_t taddr_s;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int n_items = *n_items_p;
    if (threadIdx.x == 0) {
        for (int i = 0; i < kStages; i++) {
            mbar_init(&full[i], 1 + 128);
            mbar_init(&empty[i], 1);
        }
        for (int i = 0; i < 2; i++) {
            mbar_init(&tfull[i], 1);
            mbar_init(&tempty[i], 4);
        }
        fence_mbar_init();
    }
    if (warp == 1) {
        tmem_alloc(&taddr_s, kCols < 32 ? 32 : kCols);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = taddr_s;

    if (warp == 0) {
        if (lane == 0) {
            int it = 0;
            for (int wi = blockIdx.x; wi < n_items; wi += gridDim.x) {
                const WorkItem w = items[wi];
                for (int kc = 0; kc < nk; kc++, it++) {
                    const int s = it % kStages;
                    unsigned char* st = smem + (size_t)s * kStage;
                    if (it >= kStages) mbar_wait(&empty[s], (uint32_t)((it / kStages) - 1) & 1u, status, lim);
                    mbar_arrive_expect_tx(&full[s], (uint32_t)kTileB);
                    if (NB == 128) {
                        tma_load_2d(st + kTileBytesA, &map_wg, kc * 64, w.e * 64, &full[s]);
                        tma_load_2d(st + kTileBytesA + 64 * 128, &map_wu, kc * 64, w.e * 64, &full[s]);
                    } else {
                        tma_load_2d(st + kTileBytesA, &map_wu, kc * 64, w.e * 64, &full[s]);
                    }
                }
            }
        }
        __syncwarp();
    } else if (warp >= 6) {
        // token-row gather; rows past the item's count are not copied (their
        // accumulator rows are never stored)
        const int row = (warp - 6) * 32 + lane;
        const uint32_t swz = (uint32_t)(row & 7);
        int it = 0;
        for (int wi = blockIdx.x; wi < n_items; wi += gridDim.x) {
            const WorkItem w = items[wi];
            const bool live = row < w.cnt;
            const __nv_bfloat16* src = x + (size_t)(live ? perm_token[w.a0 + row] : 0) * d;
            for (int kc = 0; kc < nk; kc++, it++) {
                const int s = it % kStages;
                if (lane == 0 && it >= kStages) mbar_wait(&empty[s], (uint32_t)((it / kStages) - 1) & 1u, status, lim);
                __syncwarp();
                unsigned char* dst = smem + (size_t)s * kStage + row * 128;
                const int c0 = kc * 64;
                if (live) {
#pragma unroll
                    for (int c = 0; c < 8; c++) {
                        const bool in = c0 + c * 8 < d;  // d is a multiple of 8: chunks are whole
                        cp_async_16(dst + (((uint32_t)c ^ swz) << 4), in ? src + c0 + c * 8 : src, in ? 16u : 0u);
                    }
                }
                cp_async_commit();
                if (it >= kGatherLag) {
                    cp_async_wait<kGatherLag>();
                    fence_proxy_async_smem();
                    mbar_arrive(&full[(it - kGatherLag) % kStages]);
                }
            }
        }
        cp_async_wait<0>();
        fence_proxy_async_smem();
        for (int j = it > kGatherLag ? it - kGatherLag : 0; j < it; j++) mbar_arrive(&full[j % kStages]);
    } else if (warp == 1) {
        if (lane == 0) {
            constexpr uint32_t idesc = idesc_bf16_m128(NB);
            int it = 0, acc = 0;
            for (int wi = blockIdx.x; wi < n_items; wi += gridDim.x, acc++) {
                const int a = acc & 1;
                if (acc >= 2) mbar_wait(&tempty[a], (uint32_t)((acc >> 1) - 1) & 1u, status, lim);
                tc_fence_after();
                for (int kc = 0; kc < nk; kc++, it++) {
                    const int s = it % kStages;
                    mbar_wait(&full[s], (uint32_t)(it / kStages) & 1u, status, lim);
                    tc_fence_after();
                    unsigned char* st = smem + (size_t)s * kStage;
                    umma_k64(tmem + (uint32_t)(a * NB), st, st + kTileBytesA, idesc, kc > 0);
                    umma_commit(&empty[s]);
                }
                umma_commit(&tfull[a]);
            }
        }
        __syncwarp();
    } else {
        const int q = warp & 3;
        const int row = 32 * q + lane;
        int acc = 0;
        for (int wi = blockIdx.x; wi < n_items; wi += gridDim.x, acc++) {
            const WorkItem w = items[wi];
            const int a = acc & 1;
            mbar_wait(&tfull[a], (uint32_t)(acc >> 1) & 1u, status, lim);
            tc_fence_after();
            const bool live = row < w.cnt;
            const float gw = live ? perm_gate[w.a0 + row] : 0.0f;
            const uint32_t base = tmem + ((uint32_t)(32 * q) << 16) + (uint32_t)(a * NB);
#pragma unroll 1
            for (int c = 0; c < 64; c += 32) {
                uint32_t u[32];
                tmem_ld32(base + (uint32_t)(NB == 128 ? 64 + c : c), u);
                float h[32];
                if (NB == 128) {
                    uint32_t g[32];
                    tmem_ld32(base + (uint32_t)c, g);
                    tmem_ld_wait();
#pragma unroll
                    for (int i = 0; i < 32; i++) h[i] = act_h(PP_ACT_SWIGLU, __uint_as_float(u[i]), __uint_as_float(g[i])) * gw;
                } else {
                    tmem_ld_wait();
#pragma unroll
                    for (int i = 0; i < 32; i++) h[i] = act_h(act, __uint_as_float(u[i]), 0.0f) * gw;
                }
                if (live) {
                    uint4* dst = reinterpret_cast<uint4*>(H + (size_t)(w.a0 + row) * 64 + c);
#pragma unroll
                    for (int v = 0; v < 4; v++)
                        dst[v] = make_uint4(pack_bf16x2(h[8 * v], h[8 * v + 1]), pack_bf16x2(h[8 * v + 2], h[8 * v + 3]),
                                            pack_bf16x2(h[8 * v + 4], h[8 * v + 5]), pack_bf16x2(h[8 * v + 6], h[8 * v + 7]));
                }
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&tempty[a]);
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 1) tmem_dealloc(tmem, kCols < 32 ? 32 : kCols);
}

PP_DEVINL bool jt_first_overflow(const WorkItem& w, long long ycap) { return (long long)w.a0 + w.cnt > ycap; }

// ============================================================== grouped down
// Persistent over (work item, column part) pairs: the njt 256-wide slices of
// d are cut into nsub parts (more, smaller tasks than items when a batch is
// small, so that every SM streams W_down); per task the H tile is loaded
// once and the part's slices stream through the B ring.  Two 256-column
// TMEM accumulators overlap the reduction epilogue with the next slice's
// MMAs.
__global__ void __launch_bounds__(kTcThreads, 1)
    down_gemm_kernel(const __grid_constant__ CUtensorMap map_h, const __grid_constant__ CUtensorMap map_wd,
                     const __grid_constant__ CUtensorMap map_y, const WorkItem* __restrict__ items,
                     const int* __restrict__ n_items_p,
                     const int* __restrict__ perm_token, int d, int njt, int nsub, __nv_bfloat16* Y, long long ycap,
                     float* yacc, int* overflow, unsigned* status, uint64_t lim) {
    pdl_wait();  // the previous kernel on the stream has completed (programmatic dependent launch)
    pdl_launch_dependents();
    constexpr int kStages = 4;
    constexpr int kTileB = 256 * 128;
    extern __shared__ __align__(1024) unsigned char smem_raw[];
    unsigned char* smem = reinterpret_cast<unsigned char*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);
    unsigned char* tileA = smem;
    unsigned char* ringB = smem + kTileBytesA;
    __shared__ uint64_t full[kStages], empty[kStages], tfull[2], tempty[2], afull, aempty;
    __shared__ uint32_t taddr_s;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int n_tasks = *n_items_p * nsub;
    // slices [jt0, jt1) of task v (item v / nsub, part v % nsub)
    auto slices = [&](int v, int& jt0, int& jt1) {
        const int sp = v % nsub;
        jt0 = sp * njt / nsub;
        jt1 = (sp + 1) * njt / nsub;
    };
    if (threadIdx.x == 0) {
        for (int i = 0; i < kStages; i++) {
            mbar_init(&full[i], 1);
            mbar_init(&empty[i], 1);
        }
        for (int i = 0; i < 2; i++) {
            mbar_init(&tfull[i], 1);
            mbar_init(&tempty[i], 4);
        }
        mbar_init(&afull, 1);
        mbar_init(&aempty, 1);
        fence_mbar_init();
    }
    if (warp == 1) {
        tmem_alloc(&taddr_s, 512);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = taddr_s;

    if (warp == 0) {
        if (lane == 0) {
            int it = 0, ii = 0;
            for (int v = blockIdx.x; v < n_tasks; v += gridDim.x, ii++) {
                const WorkItem w = items[v / nsub];
                int jt0, jt1;
                slices(v, jt0, jt1);
                if (ii >= 1) mbar_wait(&aempty, (uint32_t)(ii - 1) & 1u, status, lim);
                mbar_arrive_expect_tx(&afull, kTileBytesA);
                tma_load_2d(tileA, &map_h, 0, w.a0, &afull);
                for (int jt = jt0; jt < jt1; jt++, it++) {
                    const int s = it % kStages;
                    if (it >= kStages) mbar_wait(&empty[s], (uint32_t)((it / kStages) - 1) & 1u, status, lim);
                    mbar_arrive_expect_tx(&full[s], kTileB);
                    tma_load_2d(ringB + (size_t)s * kTileB, &map_wd, w.e * 64, jt * 256, &full[s]);
                }
            }
        }
        __syncwarp();
    } else if (warp == 1) {
        if (lane == 0) {
            constexpr uint32_t idesc = idesc_bf16_m128(256);
            int it = 0, acc = 0, ii = 0;
            for (int v = blockIdx.x; v < n_tasks; v += gridDim.x, ii++) {
                int jt0, jt1;
                slices(v, jt0, jt1);
                mbar_wait(&afull, (uint32_t)ii & 1u, status, lim);
                for (int jt = jt0; jt < jt1; jt++, it++, acc++) {
                    const int a = acc & 1;
                    if (acc >= 2) mbar_wait(&tempty[a], (uint32_t)((acc >> 1) - 1) & 1u, status, lim);
                    const int s = it % kStages;
                    mbar_wait(&full[s], (uint32_t)(it / kStages) & 1u, status, lim);
                    tc_fence_after();
                    umma_k64(tmem + (uint32_t)(a * 256), tileA, ringB + (size_t)s * kTileB, idesc, false);
                    umma_commit(&empty[s]);
                    umma_commit(&tfull[a]);
                }
                umma_commit(&aempty);
            }
        }
        __syncwarp();
    } else {
        const int q = warp & 3;
        const int row = 32 * q + lane;
        // this warp's staging area for bulk stores: four 64-column boxes of
        // its 32 rows in the 128-byte swizzle (conflict-free row writes)
        unsigned char* stage = smem + kTileBytesA + (size_t)kStages * kTileB + (size_t)q * 16384;
        int acc = 0;
        for (int v = blockIdx.x; v < n_tasks; v += gridDim.x) {
            const WorkItem w = items[v / nsub];
            int jt0, jt1;
            slices(v, jt0, jt1);
            const bool live = row < w.cnt;
            const bool group_live = 32 * q < w.cnt;  // any live row in this warp's 32 rows
            // all 32 rows live and inside Y: the group's rows go out as 2-D bulk stores
            const bool group_full = 32 * q + 32 <= w.cnt && (long long)w.a0 + 32 * q + 32 <= ycap;
            const long long arow = (long long)w.a0 + row;
            const bool in_buf = live && arow < ycap;
            const int tok = live && !in_buf ? perm_token[arow] : -1;
            float* yrow = tok >= 0 ? yacc + (size_t)tok * d : nullptr;
            if (tok >= 0 && jt_first_overflow(w, ycap)) *overflow = 1;
            __nv_bfloat16* Yrow = in_buf ? Y + (size_t)arow * d : nullptr;
            for (int jt = jt0; jt < jt1; jt++, acc++) {
                const int a = acc & 1;
                mbar_wait(&tfull[a], (uint32_t)(acc >> 1) & 1u, status, lim);
                tc_fence_after();
                const uint32_t base = tmem + ((uint32_t)(32 * q) << 16) + (uint32_t)(a * 256);
                if (group_full) {
                    // two halves of 128 columns; a half's two boxes are rewritten
                    // only after the store that last used them has read them
#pragma unroll 1
                    for (int h = 0; h < 2; h++) {
                        if (lane == 0) bulk_wait_read<1>();
                        __syncwarp();
#pragma unroll 1
                        for (int c = 128 * h; c < 128 * h + 128; c += 32) {
                            uint32_t r[32];
                            tmem_ld32(base + (uint32_t)c, r);
                            tmem_ld_wait();
#pragma unroll
                            for (int vv = 0; vv < 4; vv++) {
                                const int j = (c >> 3) + vv;  // 16-byte chunk of the 256 columns
                                const uint32_t off = (uint32_t)(j >> 3) * 4096u + (uint32_t)lane * 128u +
                                                     ((((uint32_t)j & 7u) ^ ((uint32_t)lane & 7u)) << 4);
                                *reinterpret_cast<uint4*>(stage + off) = make_uint4(
                                    pack_bf16x2(__uint_as_float(r[8 * vv]), __uint_as_float(r[8 * vv + 1])),
                                    pack_bf16x2(__uint_as_float(r[8 * vv + 2]), __uint_as_float(r[8 * vv + 3])),
                                    pack_bf16x2(__uint_as_float(r[8 * vv + 4]), __uint_as_float(r[8 * vv + 5])),
                                    pack_bf16x2(__uint_as_float(r[8 * vv + 6]), __uint_as_float(r[8 * vv + 7])));
                            }
                        }
                        fence_proxy_async_smem();
                        __syncwarp();
                        if (lane == 0) {
                            for (int b = 2 * h; b < 2 * h + 2; b++)
                                if (jt * 256 + b * 64 < d)
                                    tma_store_2d(&map_y, stage + b * 4096, jt * 256 + b * 64, w.a0 + 32 * q);
                            bulk_commit();
                        }
                    }
                }
#pragma unroll 1
                for (int c = 0; c < (group_live && !group_full ? 256 : 0); c += 32) {
                    uint32_t r[32];
                    tmem_ld32(base + (uint32_t)c, r);
                    tmem_ld_wait();
                    const int j0 = jt * 256 + c;
                    if (Yrow) {
#pragma unroll
                        for (int v = 0; v < 4; v++)
                            if (j0 + 8 * v < d)
                                *reinterpret_cast<uint4*>(Yrow + j0 + 8 * v) = make_uint4(
                                    pack_bf16x2(__uint_as_float(r[8 * v]), __uint_as_float(r[8 * v + 1])),
                                    pack_bf16x2(__uint_as_float(r[8 * v + 2]), __uint_as_float(r[8 * v + 3])),
                                    pack_bf16x2(__uint_as_float(r[8 * v + 4]), __uint_as_float(r[8 * v + 5])),
                                    pack_bf16x2(__uint_as_float(r[8 * v + 6]), __uint_as_float(r[8 * v + 7])));
                    } else if (yrow) {
#pragma unroll
                        for (int v = 0; v < 8; v++)
                            if (j0 + 4 * v < d)
                                red_add_v4(yrow + j0 + 4 * v, __uint_as_float(r[4 * v]), __uint_as_float(r[4 * v + 1]),
                                           __uint_as_float(r[4 * v + 2]), __uint_as_float(r[4 * v + 3]));
                    }
                }
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive(&tempty[a]);
            }
        }
        if (lane == 0) bulk_wait_all();  // the stores are done before the CTA's shared memory goes away
        __syncwarp();
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 1) tmem_dealloc(tmem, 512);
}

// ========================================================== small batches
// Operand-swapped grouped GEMMs for items of at most kSwN tokens (batches of
// up to kSwapMaxT tokens, where an expert sees a few tokens): the weights are the
// M = 128 operand and the item's tokens the N = kSwN operand.  A pipeline
// stage is then 16 KB of weights + 2 KB of token rows (a 128-token tile would
// spend half of every stage on padding rows), so about twice as many weight
// bytes are in flight per SM.
constexpr int kSwN = 16;
constexpr int kSwapMaxT = 128;  // batches above this keep 128-row items (experts see more tokens)
constexpr int kSwTileW = 128 * 128;   // 128 weight rows x 64 bf16
constexpr int kSwTileX = kSwN * 128;  // kSwN token rows x 64 bf16

// Gate/up (SwiGLU): D[128 x kSwN] = [64 gate rows; 64 up rows of expert e]
// . x_tokens^T over K = d.  TMEM lanes 0-63 hold the gate sums of neurons
// 0-63, lanes 64-127 the up sums; the warps reading the up lanes hand them to
// the gate warps through shared memory, which write h = silu(g) * u * gate.
__global__ void __launch_bounds__(kTcThreads, 1)
    gu_swap_kernel(const __grid_constant__ CUtensorMap map_x1, const __grid_constant__ CUtensorMap map_wg,
                   const __grid_constant__ CUtensorMap map_wu, const WorkItem* __restrict__ items,
                   const int* __restrict__ n_items_p, const int* __restrict__ perm_token,
                   const float* __restrict__ perm_gate, int nk, __nv_bfloat16* H, unsigned* status, uint64_t lim) {
    pdl_wait();  // the previous kernel on the stream has completed (programmatic dependent launch)
    pdl_launch_dependents();
    constexpr int kStages = 11;
    constexpr int kStage = kSwTileW + kSwTileX;  // 18 KB, a multiple of 1024
    extern __shared__ __align__(1024) unsigned char smem_raw[];
    unsigned char* smem = reinterpret_cast<unsigned char*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);
    __shared__ uint64_t full[kStages], empty[kStages], tfull[2], tempty[2];
    __shared__ uint32_t taddr_s;
    __shared__ float up_s[2][32][kSwN + 1];  // up sums of neurons 0-31 / 32-63 for the gate warps
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int n_items = *n_items_p;
    if (threadIdx.x == 0) {
        for (int i = 0; i < kStages; i++) {
            mbar_init(&full[i], 1);
            mbar_init(&empty[i], 1);
        }
        for (int i = 0; i < 2; i++) {
            mbar_init(&tfull[i], 1);
            mbar_init(&tempty[i], 4);
        }
        fence_mbar_init();
    }
    if (warp == 1) {
        tmem_alloc(&taddr_s, 32);  // two kSwN-column accumulators
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = taddr_s;

    if (warp == 0) {
        int it = 0;
        // the next item and its token rows are read one item ahead
        WorkItem wn = blockIdx.x < n_items ? items[blockIdx.x] : WorkItem{0, 0, 1, 0};
        int tokn = blockIdx.x < n_items ? perm_token[wn.a0 + min(lane & (kSwN - 1), wn.cnt - 1)] : 0;
        for (int wi = blockIdx.x; wi < n_items; wi += gridDim.x) {
            const WorkItem w = wn;
            // lane i < kSwN: the item's i-th token row (padding repeats the last)
            const int tok = tokn;
            if (wi + (int)gridDim.x < n_items) {
                wn = items[wi + gridDim.x];
                tokn = perm_token[wn.a0 + min(lane & (kSwN - 1), wn.cnt - 1)];
            }
            const int ng = (w.cnt + 3) >> 2;  // gather4 groups of live rows
            const int r0 = __shfl_sync(kFull, tok, (4 * lane) & 31), r1 = __shfl_sync(kFull, tok, (4 * lane + 1) & 31);
            const int r2 = __shfl_sync(kFull, tok, (4 * lane + 2) & 31), r3 = __shfl_sync(kFull, tok, (4 * lane + 3) & 31);
            for (int kc = 0; kc < nk; kc++, it++) {
                const int s = it % kStages;
                unsigned char* st = smem + (size_t)s * kStage;
                if (lane == 0) {
                    if (it >= kStages) mbar_wait(&empty[s], (uint32_t)((it / kStages) - 1) & 1u, status, lim);
                    mbar_arrive_expect_tx(&full[s], (uint32_t)(kSwTileW + ng * 512));
                }
                __syncwarp();
                if (lane < ng) tma_gather4(st + kSwTileW + lane * 512, &map_x1, kc * 64, r0, r1, r2, r3, &full[s]);
                if (lane == 0) {
                    tma_load_2d(st, &map_wg, kc * 64, w.e * 64, &full[s]);
                    tma_load_2d(st + 64 * 128, &map_wu, kc * 64, w.e * 64, &full[s]);
                }
            }
        }
        __syncwarp();
    } else if (warp == 1) {
        if (lane == 0) {
            constexpr uint32_t idesc = idesc_bf16_m128(kSwN);
            int it = 0, acc = 0;
            for (int wi = blockIdx.x; wi < n_items; wi += gridDim.x, acc++) {
                const int a = acc & 1;
                if (acc >= 2) mbar_wait(&tempty[a], (uint32_t)((acc >> 1) - 1) & 1u, status, lim);
                tc_fence_after();
                for (int kc = 0; kc < nk; kc++, it++) {
                    const int s = it % kStages;
                    mbar_wait(&full[s], (uint32_t)(it / kStages) & 1u, status, lim);
                    tc_fence_after();
                    unsigned char* st = smem + (size_t)s * kStage;
                    umma_k64(tmem + (uint32_t)(a * kSwN), st, st + kSwTileW, idesc, kc > 0);
                    umma_commit(&empty[s]);
                }
                umma_commit(&tfull[a]);
            }
        }
        __syncwarp();
    } else {
        const int q = warp & 3;  // TMEM lanes 32 q .. 32 q + 31
        int acc = 0;
        for (int wi = blockIdx.x; wi < n_items; wi += gridDim.x, acc++) {
            const WorkItem w = items[wi];
            const int a = acc & 1;
            const float gw_l = lane < w.cnt ? perm_gate[w.a0 + lane] : 0.0f;  // gate weight of token `lane`
            mbar_wait(&tfull[a], (uint32_t)(acc >> 1) & 1u, status, lim);
            tc_fence_after();
            uint32_t v[kSwN];
            tmem_ld16(tmem + ((uint32_t)(32 * q) << 16) + (uint32_t)(a * kSwN), v);
            tmem_ld_wait();
            if (q >= 2) {
#pragma unroll
                for (int t = 0; t < kSwN; t++) up_s[q - 2][lane][t] = __uint_as_float(v[t]);
            }
            named_bar_sync(1, 128);
            if (q < 2) {
                const int n = 32 * q + lane;  // this lane's neuron
#pragma unroll
                for (int t = 0; t < kSwN; t++) {
                    const float gw = __shfl_sync(kFull, gw_l, t);
                    if (t < w.cnt) {
                        const float h = act_h(PP_ACT_SWIGLU, up_s[q][lane][t], __uint_as_float(v[t])) * gw;
                        H[(size_t)(w.a0 + t) * 64 + n] = __float2bfloat16_rn(h);
                    }
                }
            }
            named_bar_sync(1, 128);  // up_s is free for the next item
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&tempty[a]);
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 1) tmem_dealloc(tmem, 32);
}

// Down projection: per task (item, part of the ceil(d / 128) row tiles),
// D[128 x kSwN] = W_down[128 rows, 64 columns of expert e] . H_item^T; the
// item's kSwN H rows stay in shared memory for the task while the W_down
// tiles stream through the ring (two H buffers, so that the next task's
// tiles follow without a gap).  Lane = output row, column t = token: Y row
// a0 + t (or, past ycap, a reduction into yacc) receives it.
__global__ void __launch_bounds__(kTcThreads, 1)
    down_swap_kernel(const __grid_constant__ CUtensorMap map_h, const __grid_constant__ CUtensorMap map_wd,
                     const WorkItem* __restrict__ items, const int* __restrict__ n_items_p,
                     const int* __restrict__ perm_token, int d, int nrt, int nsub, __nv_bfloat16* Y, long long ycap,
                     float* yacc, int* overflow, unsigned* status, uint64_t lim) {
    pdl_wait();  // the previous kernel on the stream has completed (programmatic dependent launch)
    pdl_launch_dependents();
    constexpr int kStages = 12;
    extern __shared__ __align__(1024) unsigned char smem_raw[];
    unsigned char* smem = reinterpret_cast<unsigned char*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);
    unsigned char* tileH = smem;                // 2 x kSwTileX bytes (1024-aligned)
    unsigned char* ring = smem + 2 * 2048;      // kStages x kSwTileW
    __shared__ uint64_t full[kStages], empty[kStages], tfull[2], tempty[2], hfull[2], hempty[2];
    __shared__ uint32_t taddr_s;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int n_tasks = *n_items_p * nsub;
    auto tiles = [&](int v, int& r0, int& r1) {  // row tiles [r0, r1) of task v
        const int sp = v % nsub;
        r0 = sp * nrt / nsub;
        r1 = (sp + 1) * nrt / nsub;
    };
    if (threadIdx.x == 0) {
        for (int i = 0; i < kStages; i++) {
            mbar_init(&full[i], 1);
            mbar_init(&empty[i], 1);
        }
        for (int i = 0; i < 2; i++) {
            mbar_init(&tfull[i], 1);
            mbar_init(&tempty[i], 4);
        }
        for (int i = 0; i < 2; i++) {
            mbar_init(&hfull[i], 1);
            mbar_init(&hempty[i], 1);
        }
        fence_mbar_init();
    }
    if (warp == 1) {
        tmem_alloc(&taddr_s, 32);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = taddr_s;

    if (warp == 0) {
        if (lane == 0) {
            int it = 0, ii = 0;
            WorkItem wn = blockIdx.x < n_tasks ? items[blockIdx.x / nsub] : WorkItem{0, 0, 0, 0};
            for (int v = blockIdx.x; v < n_tasks; v += gridDim.x, ii++) {
                const WorkItem w = wn;
                if (v + (int)gridDim.x < n_tasks) wn = items[(v + gridDim.x) / nsub];  // next task's item, early
                int r0, r1;
                tiles(v, r0, r1);
                const int hb = ii & 1;
                if (ii >= 2) mbar_wait(&hempty[hb], (uint32_t)((ii >> 1) - 1) & 1u, status, lim);
                mbar_arrive_expect_tx(&hfull[hb], kSwTileX);
                tma_load_2d(tileH + hb * 2048, &map_h, 0, w.a0, &hfull[hb]);
                for (int rt = r0; rt < r1; rt++, it++) {
                    const int s = it % kStages;
                    if (it >= kStages) mbar_wait(&empty[s], (uint32_t)((it / kStages) - 1) & 1u, status, lim);
                    mbar_arrive_expect_tx(&full[s], kSwTileW);
                    tma_load_2d(ring + (size_t)s * kSwTileW, &map_wd, w.e * 64, rt * 128, &full[s]);
                }
            }
        }
        __syncwarp();
    } else if (warp == 1) {
        if (lane == 0) {
            constexpr uint32_t idesc = idesc_bf16_m128(kSwN);
            int it = 0, acc = 0, ii = 0;
            for (int v = blockIdx.x; v < n_tasks; v += gridDim.x, ii++) {
                int r0, r1;
                tiles(v, r0, r1);
                const int hb = ii & 1;
                mbar_wait(&hfull[hb], (uint32_t)(ii >> 1) & 1u, status, lim);
                for (int rt = r0; rt < r1; rt++, it++, acc++) {
                    const int a = acc & 1;
                    if (acc >= 2) mbar_wait(&tempty[a], (uint32_t)((acc >> 1) - 1) & 1u, status, lim);
                    const int s = it % kStages;
                    mbar_wait(&full[s], (uint32_t)(it / kStages) & 1u, status, lim);
                    tc_fence_after();
                    umma_k64(tmem + (uint32_t)(a * kSwN), ring + (size_t)s * kSwTileW, tileH + hb * 2048, idesc,
                             false);
                    umma_commit(&empty[s]);
                    umma_commit(&tfull[a]);
                }
                umma_commit(&hempty[hb]);
            }
        }
        __syncwarp();
    } else {
        const int q = warp & 3;
        int acc = 0;
        for (int v = blockIdx.x; v < n_tasks; v += gridDim.x) {
            const WorkItem w = items[v / nsub];
            int r0, r1;
            tiles(v, r0, r1);
            // token of assignment row a0 + lane (for rows past ycap)
            const long long arow_l = (long long)w.a0 + lane;
            const int tok_l = lane < w.cnt && arow_l >= ycap ? perm_token[arow_l] : -1;
            const bool spill = (long long)w.a0 + w.cnt > ycap;  // some of the item's rows go to yacc
            if (lane == 0 && spill) *overflow = 1;
            for (int rt = r0; rt < r1; rt++, acc++) {
                const int a = acc & 1;
                mbar_wait(&tfull[a], (uint32_t)(acc >> 1) & 1u, status, lim);
                tc_fence_after();
                uint32_t val[kSwN];
                tmem_ld16(tmem + ((uint32_t)(32 * q) << 16) + (uint32_t)(a * kSwN), val);
                tmem_ld_wait();
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive(&tempty[a]);
                const int row = rt * 128 + 32 * q + lane;  // output element of d
                if (!spill) {  // every row of the item is kept: only its cnt columns are stored
                    if (row < d) {
                        __nv_bfloat16* yp = Y + (size_t)w.a0 * d + row;
#pragma unroll
                        for (int t = 0; t < kSwN; t++) {
                            if (t >= w.cnt) break;
                            yp[(size_t)t * d] = __float2bfloat16_rn(__uint_as_float(val[t]));
                        }
                    }
                } else {
#pragma unroll
                    for (int t = 0; t < kSwN; t++) {
                        const int tk = __shfl_sync(kFull, tok_l, t);
                        if (t < w.cnt && row < d) {
                            const long long arow = (long long)w.a0 + t;
                            if (arow < ycap)
                                Y[(size_t)arow * d + row] = __float2bfloat16_rn(__uint_as_float(val[t]));
                            else
                                atomicAdd(&yacc[(size_t)tk * d + row], __uint_as_float(val[t]));
                        }
                    }
                }
            }
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 1) tmem_dealloc(tmem, 32);
}

// =================================================================== combine
// y[t] = the sum of token t's assignment rows Y[pos] in ascending expert
// order, plus yacc[t] when the down projection overflowed (yacc is then
// cleared again).  Grid (T, ceil(d / 1024)): 128 threads of 8 columns each.
// The expert list is built in parallel: 128 experts per round, compacted in
// ascending order with ballots.
__global__ void __launch_bounds__(128) combine_kernel(const uint32_t* __restrict__ bits, const int* __restrict__ invpos,
                                                      const __nv_bfloat16* __restrict__ Y, long long ycap,
                                                      float* yacc, const int* __restrict__ overflow, int T, int E,
                                                      int d, __nv_bfloat16* y) {
    pdl_wait();  // the previous kernel on the stream has completed (programmatic dependent launch)
    pdl_launch_dependents();
    const int t = blockIdx.x, tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    __shared__ int pos_s[kMaxExperts];
    __shared__ int wn_s[4];
    int n = 0;
    for (int e0 = 0; e0 < E; e0 += 128) {
        const int e = e0 + tid;
        bool on = e < E && ((bits[(size_t)t * 8 + (e >> 5)] >> (e & 31)) & 1u);
        const int pos = on ? invpos[(size_t)t * E + e] : 0;
        on = on && pos < ycap;
        const unsigned bal = __ballot_sync(kFull, on);
        if (lane == 0) wn_s[warp] = __popc(bal);
        __syncthreads();
        int base = n;
        for (int w = 0; w < warp; w++) base += wn_s[w];
        if (on) pos_s[base + __popc(bal & ((1u << lane) - 1u))] = pos;
        n += wn_s[0] + wn_s[1] + wn_s[2] + wn_s[3];
        __syncthreads();
    }
    const int c = blockIdx.y * 1024 + tid * 8;
    if (c >= d) return;
    float acc[8] = {0, 0, 0, 0, 0, 0, 0, 0};
    if (*overflow != 0) {
        float4* ya = reinterpret_cast<float4*>(yacc + (size_t)t * d + c);
        const float4 a0 = ya[0], a1 = ya[1];
        acc[0] = a0.x; acc[1] = a0.y; acc[2] = a0.z; acc[3] = a0.w;
        acc[4] = a1.x; acc[5] = a1.y; acc[6] = a1.z; acc[7] = a1.w;
        ya[0] = make_float4(0.f, 0.f, 0.f, 0.f);  // keep the accumulator zero at rest
        ya[1] = make_float4(0.f, 0.f, 0.f, 0.f);
    }
    // rows added in ascending expert order; their loads go out 4 at a time
    for (int i0 = 0; i0 < n; i0 += 4) {
        uint4 v4[4];
#pragma unroll
        for (int u = 0; u < 4; u++)
            if (i0 + u < n) v4[u] = *reinterpret_cast<const uint4*>(Y + (size_t)pos_s[i0 + u] * d + c);
#pragma unroll
        for (int u = 0; u < 4; u++) {
            if (i0 + u >= n) break;
            const uint4 v = v4[u];
            acc[0] += bf16lo(v.x); acc[1] += bf16hi(v.x); acc[2] += bf16lo(v.y); acc[3] += bf16hi(v.y);
            acc[4] += bf16lo(v.z); acc[5] += bf16hi(v.z); acc[6] += bf16lo(v.w); acc[7] += bf16hi(v.w);
        }
    }
    *reinterpret_cast<uint4*>(y + (size_t)t * d + c) =
        make_uint4(pack_bf16x2(acc[0], acc[1]), pack_bf16x2(acc[2], acc[3]), pack_bf16x2(acc[4], acc[5]),
                   pack_bf16x2(acc[6], acc[7]));
}

// ====================================================================== host
namespace {

// Launch with programmatic dependent launch allowed: the kernel may be
// scheduled while its predecessor on the stream finishes, and waits for it
// in griddepcontrol.wait (pdl_wait) before touching memory.
template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(void (*kern)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t st, Args&&... args) {
    cudaLaunchConfig_t cfg{};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    cudaError_t e = cudaLaunchKernelEx(&cfg, kern, std::forward<Args>(args)...);
    if (e == cudaErrorNotSupported) {
        (void)cudaGetLastError();
        cfg.numAttrs = 0;
        e = cudaLaunchKernelEx(&cfg, kern, std::forward<Args>(args)...);
    }
    return e;
}

// Launch through launch_pdl; returns the error from the enclosing function.
#define PP_LAUNCH(...)                                   \
    do {                                                 \
        const cudaError_t le_ = launch_pdl(__VA_ARGS__); \
        if (le_ != cudaSuccess) return le_;              \
    } while (0)


// bf16 [outer][inner] row-major, SW128 boxes.  `promote` is the L2 fill
// granularity: 256 B where the neighbouring 128 B of a row is read next by
// the same CTA (K-major operand streams), 128 B where it belongs to another
// expert that may not be selected (the 64-column blocks of W_down).
bool encode_2d(CUtensorMap* map, const void* base, uint64_t inner, uint64_t outer, uint32_t box_inner,
               uint32_t box_outer, CUtensorMapL2promotion promote = CU_TENSOR_MAP_L2_PROMOTION_L2_256B) {
    auto enc = tensor_map_encoder();
    if (!enc) return false;
    const cuuint64_t dims[2] = {inner, outer};
    const cuuint64_t strides[1] = {inner * 2};
    const cuuint32_t box[2] = {box_inner, box_outer};
    const cuuint32_t estr[2] = {1, 1};
    return enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, estr,
               CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, promote,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

template <typename K>
cudaError_t set_smem(K kern, size_t bytes) {
    return cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)bytes);
}

int router_ne(int E) { return E <= 32 ? 32 : E <= 64 ? 64 : E <= 128 ? 128 : E <= 160 ? 160 : E <= 192 ? 192 : E <= 224 ? 224 : 256; }

template <int NE>
cudaError_t launch_router(const CUtensorMap& mx, const CUtensorMap& mwr, int T, int E, int nk, int kpb, int nsplit,
                          float* part, unsigned* status, uint64_t lim, cudaStream_t st) {
    const size_t smem = 4 * (size_t)(kTileBytesA + NE * 128) + 1024;
    cudaError_t e = set_smem(router_gemm_kernel<NE>, smem);
    if (e != cudaSuccess) return e;
    PP_LAUNCH(router_gemm_kernel<NE>, dim3((T + 127) / 128, nsplit), dim3(kTcThreads), smem, st, mx, mwr, T, E, nk,
        kpb, part, status, lim);
    return cudaGetLastError();
}

}  // namespace

GroupedPlan grouped_plan(int T, int d, int E, int sms) {
    GroupedPlan g{};
    g.nk = (d + 63) / 64;  // the last chunk's columns past d are zero-filled by TMA
    // router K splits: at most one wave of CTAs, at least 4 chunks each
    const int mt = (T + 127) / 128;
    const int ns = std::max(1, std::min(sms / mt, std::min(g.nk / 4, 64)));
    g.kpb = (g.nk + ns - 1) / ns;
    g.nsplit = (g.nk + g.kpb - 1) / g.kpb;
    const int rows = T <= kSwapMaxT ? kSwN : 128;  // rows per work item
    g.max_items = (int)std::min<long long>((long long)T * E / rows + E + 1, (long long)T * E);
    g.nnz_max = (long long)T * E;
    g.ycap = (long long)T * std::min(E, 64);  // assignment rows kept for the combine
    return g;
}

cudaError_t grouped_route(const GroupedArgs& a, cudaStream_t st) {
    const GroupedPlan& g = a.plan;
    CUtensorMap mx, mwr;
    const int NE = router_ne(a.E);
    if (!encode_2d(&mx, a.x, a.d, a.T, 64, 128) || !encode_2d(&mwr, a.Wr, a.d, a.E, 64, NE)) return cudaErrorInvalidValue;
    cudaError_t e;
    switch (NE) {
        case 32: e = launch_router<32>(mx, mwr, a.T, a.E, g.nk, g.kpb, g.nsplit, a.part, a.status, a.timeout_ns, st); break;
        case 64: e = launch_router<64>(mx, mwr, a.T, a.E, g.nk, g.kpb, g.nsplit, a.part, a.status, a.timeout_ns, st); break;
        case 128: e = launch_router<128>(mx, mwr, a.T, a.E, g.nk, g.kpb, g.nsplit, a.part, a.status, a.timeout_ns, st); break;
        case 160: e = launch_router<160>(mx, mwr, a.T, a.E, g.nk, g.kpb, g.nsplit, a.part, a.status, a.timeout_ns, st); break;
        case 192: e = launch_router<192>(mx, mwr, a.T, a.E, g.nk, g.kpb, g.nsplit, a.part, a.status, a.timeout_ns, st); break;
        case 224: e = launch_router<224>(mx, mwr, a.T, a.E, g.nk, g.kpb, g.nsplit, a.part, a.status, a.timeout_ns, st); break;
        default: e = launch_router<256>(mx, mwr, a.T, a.E, g.nk, g.kpb, g.nsplit, a.part, a.status, a.timeout_ns, st); break;
    }
    if (e != cudaSuccess) return e;
    if ((a.rule == PP_SEL_MIN_PREFIX || a.rule == PP_SEL_PAPER) && a.p < 1.0f) {
        PP_LAUNCH(select_part_cut_kernel, dim3(a.T), dim3(256), 0, st, a.part, g.nsplit, a.T, a.E, a.p, a.rule,
                  a.gate, a.ids, a.counts, a.gates, a.logits_out, a.status);
        return cudaGetLastError();
    }
    if (a.T <= kCtaSelectMaxTokens) {
        PP_LAUNCH(select_part_cta_kernel, dim3(a.T), dim3(256), 0, st, a.part, g.nsplit, a.T, a.E, a.p, a.rule,
            a.gate, a.ids, a.counts, a.gates, a.logits_out, a.status);
        return cudaGetLastError();
    }
    const dim3 grid((a.T + 7) / 8), block(256);
    switch (sel_slots_for(a.E)) {
        case 1: PP_LAUNCH(select_part_kernel<1>, dim3(grid), dim3(block), 0, st, a.part, g.nsplit, a.T, a.E, a.p, a.rule,
                a.gate, a.ids, a.counts, a.gates, a.logits_out, a.status); break;
        case 2: PP_LAUNCH(select_part_kernel<2>, dim3(grid), dim3(block), 0, st, a.part, g.nsplit, a.T, a.E, a.p, a.rule,
                a.gate, a.ids, a.counts, a.gates, a.logits_out, a.status); break;
        case 4: PP_LAUNCH(select_part_kernel<4>, dim3(grid), dim3(block), 0, st, a.part, g.nsplit, a.T, a.E, a.p, a.rule,
                a.gate, a.ids, a.counts, a.gates, a.logits_out, a.status); break;
        default: PP_LAUNCH(select_part_kernel<8>, dim3(grid), dim3(block), 0, st, a.part, g.nsplit, a.T, a.E, a.p, a.rule,
                a.gate, a.ids, a.counts, a.gates, a.logits_out, a.status); break;
    }
    return cudaGetLastError();
}

cudaError_t grouped_ffn(const GroupedArgs& a, int sms, cudaStream_t st) {
    const GroupedPlan& g = a.plan;
    const bool gated = a.act == PP_ACT_SWIGLU;
    cudaError_t e;
    // dispatch
    if (a.T <= kSmallDispatchMaxT) {
        PP_LAUNCH(dispatch_small_kernel, dim3(1), dim3(1024), 0, st, a.ids, a.counts, a.gates, a.T, a.E, a.bits,
            a.offsets, reinterpret_cast<WorkItem*>(a.items), a.n_items, a.perm_token, a.perm_gate, a.invpos,
            a.overflow, a.T <= kSwapMaxT ? kSwN : 128, a.status);
    } else {
        const int nblk = (a.T + kDispBlock - 1) / kDispBlock;
        PP_LAUNCH(dispatch_bits_kernel, dim3((a.T + 7) / 8), dim3(256), 0, st, a.ids, a.counts, a.gates, a.T, a.E,
            a.bits, a.gexp, a.status);
        PP_LAUNCH(dispatch_count_kernel, dim3(nblk), dim3(kDispBlock), 0, st, a.bits, a.T, a.E, a.wcnt, a.blkcnt);
        PP_LAUNCH(dispatch_scan_kernel, dim3(1), dim3(kMaxExperts), 0, st, a.blkcnt, nblk, a.E, a.offsets, a.blkbase,
            reinterpret_cast<WorkItem*>(a.items), a.n_items, a.overflow);
        PP_LAUNCH(dispatch_scatter_kernel, dim3(nblk, std::min(8, a.E)), dim3(kDispBlock), 0, st, a.bits, a.gexp, a.T, a.E, a.wcnt,
            a.blkbase, a.perm_token, a.perm_gate, a.invpos);
    }
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    // grouped gate/up
    CUtensorMap mx1, mwg, mwu, mh, mwd;
    if (!encode_2d(&mx1, a.x, a.d, a.T, 64, 1) || !encode_2d(&mwu, a.Wu, a.d, (uint64_t)a.E * 64, 64, 64) ||
        !encode_2d(&mwg, gated ? a.Wg : a.Wu, a.d, (uint64_t)a.E * 64, 64, 64) ||
        !encode_2d(&mh, a.H, 64, (uint64_t)g.nnz_max + 128, 64, 128) ||
        !encode_2d(&mwd, a.Wd, (uint64_t)a.E * 64, a.d, 64, 256, CU_TENSOR_MAP_L2_PROMOTION_L2_128B))
        return cudaErrorInvalidValue;
    const int grid = std::max(1, std::min(sms, g.max_items));
    const WorkItem* items = reinterpret_cast<const WorkItem*>(a.items);
    // batches of up to kSwapMaxT tokens: items of at most kSwN rows and the
    // operand-swapped kernels (weights as the M = 128 operand)
    const bool small = a.T <= kSwapMaxT;
    if (gated && small) {
        const size_t smem = 11 * (size_t)(kSwTileW + kSwTileX) + 1024;
        if ((e = set_smem(gu_swap_kernel, smem)) != cudaSuccess) return e;
        PP_LAUNCH(gu_swap_kernel, dim3(grid), dim3(kTcThreads), smem, st, mx1, mwg, mwu, items, a.n_items,
            a.perm_token, a.perm_gate, g.nk, a.H, a.status, a.timeout_ns);
    } else if (gated) {
        const size_t smem = 6 * (size_t)(kTileBytesA + 128 * 128) + 1024;
        if ((e = set_smem(gu_gemm_kernel<128>, smem)) != cudaSuccess) return e;
        PP_LAUNCH(gu_gemm_kernel<128>, dim3(grid), dim3(kGuThreads), smem, st,
            reinterpret_cast<const __nv_bfloat16*>(a.x), a.d, mwg, mwu, items, a.n_items, a.perm_token, a.perm_gate,
            g.nk, a.act, a.H, a.status, a.timeout_ns);
    } else {
        const size_t smem = 8 * (size_t)(kTileBytesA + 64 * 128) + 1024;
        if ((e = set_smem(gu_gemm_kernel<64>, smem)) != cudaSuccess) return e;
        PP_LAUNCH(gu_gemm_kernel<64>, dim3(grid), dim3(kGuThreads), smem, st,
            reinterpret_cast<const __nv_bfloat16*>(a.x), a.d, mwg, mwu, items, a.n_items, a.perm_token, a.perm_gate,
            g.nk, a.act, a.H, a.status, a.timeout_ns);
    }
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    // grouped down + scatter-add
    if (small) {
        CUtensorMap mh16, mwd128;
        if (!encode_2d(&mh16, a.H, 64, (uint64_t)g.nnz_max + 128, 64, kSwN) ||
            !encode_2d(&mwd128, a.Wd, (uint64_t)a.E * 64, a.d, 64, 128, CU_TENSOR_MAP_L2_PROMOTION_L2_128B))
            return cudaErrorInvalidValue;
        const size_t smem = 2 * 2048 + 12 * (size_t)kSwTileW + 1024;
        if ((e = set_smem(down_swap_kernel, smem)) != cudaSuccess) return e;
        // each item's ceil(d / 128) row tiles cut into up to 4 tasks, so that
        // every SM streams W_down
        const int nrt = (a.d + 127) / 128;
        const int nsub = std::min(4, nrt);
        const int grid6 = std::max(1, (int)std::min<long long>(sms, (long long)g.max_items * nsub));
        PP_LAUNCH(down_swap_kernel, dim3(grid6), dim3(kTcThreads), smem, st, mh16, mwd128, items, a.n_items,
            a.perm_token, a.d, nrt, nsub, a.Y, g.ycap, a.yacc, a.overflow, a.status, a.timeout_ns);
        if ((e = cudaGetLastError()) != cudaSuccess) return e;
    } else {
        // A tile, the 4-stage W_down ring, 4 x 16 KB store staging
        const size_t smem = (size_t)kTileBytesA + 4 * (size_t)256 * 128 + 4 * (size_t)16384 + 1024;
        CUtensorMap my;
        if (!encode_2d(&my, a.Y, a.d, (uint64_t)g.ycap, 64, 32)) return cudaErrorInvalidValue;
        if ((e = set_smem(down_gemm_kernel, smem)) != cudaSuccess) return e;
        // up to 256 tokens: about one 128-row item per expert, fewer than the
        // SMs can share evenly, so each item's columns are cut into 4 tasks
        const int njt = (a.d + 255) / 256;
        const int nsub = a.T <= kSmallDispatchMaxT ? std::min(4, njt) : 1;
        const int grid6 = std::max(1, (int)std::min<long long>(sms, (long long)g.max_items * nsub));
        PP_LAUNCH(down_gemm_kernel, dim3(grid6), dim3(kTcThreads), smem, st, mh, mwd, my, items, a.n_items, a.perm_token,
            a.d, njt, nsub, a.Y, g.ycap, a.yacc, a.overflow, a.status, a.timeout_ns);
        if ((e = cudaGetLastError()) != cudaSuccess) return e;
    }
    PP_LAUNCH(combine_kernel, dim3(a.T, (a.d + 1023) / 1024), dim3(128), 0, st, a.bits, a.invpos, a.Y, g.ycap,
        a.yacc, a.overflow, a.T, a.E, a.d, reinterpret_cast<__nv_bfloat16*>(a.y));
    return cudaGetLastError();
}

}  // namespace pp
