// Fused decode layer for small token counts (PrunePath Sec. 3.1 end to end).
//
// One cooperative, persistent launch of one CTA per SM does, for T <= TS
// tokens:
//   phase 1  router (Eq. routing_logits): CTA b bulk-loads its rows of W_r
//            and dots them with x (fp32 FMA), writing logits to the workspace;
//   -- grid barrier --
//   select   every CTA redundantly runs the warp selection of each token
//            (Eq. softmax_prob, the descending order, Eq. tau_thresh_activate)
//            and forms U, the union of the tokens' activated experts;
//   phase 4  gate/up (Eq. ffn on the expert blocks): the U*64 neurons are
//            split evenly over the grid; each consumer warp bulk-loads the
//            gate and up rows of one neuron into its own shared-memory slot,
//            computes h = act(.) * gate weight (Eq. moe_output) per token and
//            stores it to the workspace;
//   -- grid barrier --
//   phase 6  down projection: CTA b owns R6 rows of W_down and y; a producer
//            warp streams the [R6 x 64] column block of every expert in U
//            with 2-D tensor TMA (these loads are issued before phase 4 runs,
//            so they overlap it), the consumer warps accumulate
//            y[t][row] = sum_u sum_n W_down[row][u*64+n] * h[u][t][n] in fp32
//            in registers and write y once (no atomics, deterministic).
// Only the selected expert blocks are read from HBM.
#include "pp_common.cuh"
#include "pp_select.cuh"
#include "pp_kernels.h"

namespace pp {

constexpr int kConsumerWarps = 8;
constexpr int kDecThreads = (kConsumerWarps + 1) * 32;
constexpr int kNS6 = 8;   // phase-6 ring slots
constexpr int kMaxNS4 = kConsumerWarps;

// barrier indices in the first bytes of shared memory
constexpr int kBarX = 0, kBarR = 1, kBarFull4 = 2, kBarFull6 = kBarFull4 + kMaxNS4,
              kBarEmpty6 = kBarFull6 + kNS6, kNumBars = kBarEmpty6 + kNS6;

template <typename TW, int TS, int S>
PP_DEVINL void select_tokens(const DecodeArgs& a, float* gw, unsigned* mask, bool cta0) {
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int E = a.E;
    if (warp >= a.T) return;
    const int t = warp;
    unsigned long long key[S];
    bool finite = true;
    const float* row = a.logit_ws + (size_t)t * E;
    const int k = warp_select<S>([&](int j) { return __ldcg(row + j); }, E, a.p, a.rule, key, &finite);
    if (!finite) {
        if (lane == 0) record_status(a.status, PP_ERR_NONFINITE);
    }
#pragma unroll
    for (int s = 0; s < S; s++) {
        const int r = lane * S + s;
        if (r >= E) continue;
        const bool on = finite && r < k;
        const int e = finite ? key_index(key[s]) : r;
        const float gv = on ? gate_of(a.gate, key[s]) : 0.0f;
        if (on) {
            gw[t * E + e] = gv;
            atomicOr(&mask[e], 1u << t);
        }
        if (cta0 && a.sel_ids) {
            a.sel_ids[(size_t)t * E + r] = on ? e : -1;
            a.sel_gates[(size_t)t * E + r] = gv;
        }
    }
    if (cta0) {
        if (a.sel_counts && lane == 0) a.sel_counts[t] = k;
        if (a.sel_logits)
            for (int j = lane; j < E; j += 32) a.sel_logits[(size_t)t * E + j] = __ldcg(row + j);
    }
}

// Selection given by the caller (pp_sparse_ffn): gates are summed per expert
// so repeated ids behave like repeated terms of the sum.
PP_DEVINL void load_given_selection(const DecodeArgs& a, float* gw, unsigned* mask) {
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (warp >= a.T) return;
    const int t = warp, E = a.E;
    int cnt = a.sel_counts[t];
    if (cnt < 0 || cnt > E) {
        if (lane == 0) record_status(a.status, PP_ERR_INVALID_ARG);
        cnt = cnt < 0 ? 0 : E;
    }
    for (int r = lane; r < cnt; r += 32) {
        const int e = a.sel_ids[(size_t)t * E + r];
        if (e < 0 || e >= E) {
            record_status(a.status, PP_ERR_INVALID_ARG);
            continue;
        }
        atomicAdd(&gw[t * E + e], a.sel_gates[(size_t)t * E + r]);
        atomicOr(&mask[e], 1u << t);
    }
}

template <typename TW, int TS>
__global__ void __launch_bounds__(kDecThreads, 1) decode_layer_kernel(const __grid_constant__ DecodeArgs a) {
    extern __shared__ __align__(1024) unsigned char smem[];
    using EL = Elem<TW>;
    constexpr int kEl = EL::kPer16B;
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const bool is_producer = warp == kConsumerWarps;
    const int T = a.T, d = a.d, E = a.E;
    const int G = gridDim.x, b = blockIdx.x;
    const int nchunk = d / kEl;  // 16-byte chunks per row
    const size_t rowb = (size_t)d * sizeof(TW);
    const bool gated = a.act == PP_ACT_SWIGLU;
    const uint64_t lim = a.timeout_ns;

    uint64_t* bars = reinterpret_cast<uint64_t*>(smem);
    TW* xs = reinterpret_cast<TW*>(smem + a.off_x);
    float* gw = reinterpret_cast<float*>(smem + a.off_gw);
    unsigned* mask = reinterpret_cast<unsigned*>(smem + a.off_mask);
    int* ulist = reinterpret_cast<int*>(smem + a.off_ulist);
    float* red = reinterpret_cast<float*>(smem + a.off_red);
    float* hs = reinterpret_cast<float*>(smem + a.off_h);
    unsigned char* ring4 = smem + a.off_ring4;
    unsigned char* ring6 = smem + a.off_ring6;
    __shared__ int s_nU;
    __shared__ int s_wcount[kConsumerWarps + 1];

    if (tid == 0) {
        for (int i = 0; i < kNumBars; i++)
            mbar_init(&bars[i], (i >= kBarEmpty6) ? kConsumerWarps : 1);
        fence_mbar_init();
    }
    for (int i = tid; i < TS * E; i += blockDim.x) gw[i] = 0.0f;
    for (int i = tid; i < kMaxExperts; i += blockDim.x) mask[i] = 0u;
    __syncthreads();

    // this CTA's router rows [j0, j1) of W_r (phase 1)
    const int rpc = (E + G - 1) / G;
    const int j0 = b * rpc, j1 = min(E, j0 + rpc);
    const int nrows = a.do_route ? max(0, j1 - j0) : 0;

    // x -> shared memory (all T rows are contiguous), and the router rows
    if (is_producer && lane == 0) {
        const uint32_t bytes = (uint32_t)(T * rowb);
        mbar_arrive_expect_tx(&bars[kBarX], bytes);
        bulk_g2s(xs, a.x, bytes, &bars[kBarX]);
        if (nrows > 0) {
            const TW* wr = reinterpret_cast<const TW*>(a.Wr);
            const uint32_t rbytes = (uint32_t)(nrows * rowb);
            mbar_arrive_expect_tx(&bars[kBarR], rbytes);
            bulk_g2s(ring4, wr + (size_t)j0 * d, rbytes, &bars[kBarR]);
        }
    }
    // every CTA waits for its copy of x here, so no bulk copy is ever still
    // in flight when a CTA that has no work left exits
    mbar_wait(&bars[kBarX], 0, a.status, lim);

    // ---------------------------------------------------------- phase 1
    if (a.do_route) {
        if (!is_producer && nrows > 0) {
            mbar_wait(&bars[kBarR], 0, a.status, lim);
            const TW* rows_s = reinterpret_cast<const TW*>(ring4);
            for (int r0 = 0; r0 < nrows; r0 += 2) {
                float acc[2][TS];
#pragma unroll
                for (int i = 0; i < 2; i++)
#pragma unroll
                    for (int t = 0; t < TS; t++) acc[i][t] = 0.0f;
                for (int c = tid; c < nchunk; c += kConsumerWarps * 32) {
                    float xf[TS][kEl];
#pragma unroll
                    for (int t = 0; t < TS; t++)
                        if (t < T) EL::unpack(reinterpret_cast<const uint4*>(xs + (size_t)t * d)[c], xf[t]);
#pragma unroll
                    for (int i = 0; i < 2; i++) {
                        if (r0 + i >= nrows) break;
                        float wf[kEl];
                        EL::unpack(reinterpret_cast<const uint4*>(rows_s + (size_t)(r0 + i) * d)[c], wf);
#pragma unroll
                        for (int t = 0; t < TS; t++)
                            if (t < T)
#pragma unroll
                                for (int q = 0; q < kEl; q++) acc[i][t] = fmaf(wf[q], xf[t][q], acc[i][t]);
                    }
                }
#pragma unroll
                for (int i = 0; i < 2; i++)
#pragma unroll
                    for (int t = 0; t < TS; t++) {
                        const float v = warp_sum(acc[i][t]);
                        if (lane == 0) red[(warp * 2 + i) * TS + t] = v;
                    }
                named_bar_sync(1, kConsumerWarps * 32);
                if (tid < 2 * TS) {
                    const int i = tid / TS, t = tid % TS;
                    if (r0 + i < nrows && t < T) {
                        float v = 0.0f;
                        for (int w = 0; w < kConsumerWarps; w++) v += red[(w * 2 + i) * TS + t];
                        a.logit_ws[(size_t)t * E + j0 + r0 + i] = v;
                    }
                }
                named_bar_sync(1, kConsumerWarps * 32);
            }
        }
        grid_barrier(a.bar, a.status, lim);
        if (a.sel_slots == 1) select_tokens<TW, TS, 1>(a, gw, mask, b == 0);
        else if (a.sel_slots == 2) select_tokens<TW, TS, 2>(a, gw, mask, b == 0);
        else if (a.sel_slots == 4) select_tokens<TW, TS, 4>(a, gw, mask, b == 0);
        else select_tokens<TW, TS, 8>(a, gw, mask, b == 0);
    } else {
        load_given_selection(a, gw, mask);
    }
    __syncthreads();
    if (!a.do_ffn) return;

    // union U of the tokens' activated experts, ascending expert index
    {
        const int e = tid;
        const bool on = e < E && mask[e] != 0u;
        const unsigned bal = __ballot_sync(kFull, on);
        if (lane == 0) s_wcount[warp] = __popc(bal);
        __syncthreads();
        if (tid == 0) {
            int acc = 0;
            for (int w = 0; w <= kConsumerWarps; w++) {
                const int c = s_wcount[w];
                s_wcount[w] = acc;
                acc += c;
            }
            s_nU = acc;
        }
        __syncthreads();
        if (on) ulist[s_wcount[warp] + __popc(bal & ((1u << lane) - 1u))] = e;
        __syncthreads();
    }
    const int nU = s_nU;

    // phase-6 geometry: CTA b owns rows [r0, r0 + rows) of W_down and y
    const int R6 = a.R6;
    const int r0 = b * R6;
    const int rows = max(0, min(R6, d - r0));
    const uint32_t stage6 = (uint32_t)(R6 * kDExpert * sizeof(TW));
    const int ntiles = rows > 0 ? nU : 0;

    // producer: prefetch the first phase-6 tiles now, so they stream while
    // phase 4 runs
    if (is_producer && lane == 0) {
        fence_proxy_async_smem();
        for (int u = 0; u < min(ntiles, kNS6); u++) {
            mbar_arrive_expect_tx(&bars[kBarFull6 + u], stage6);
            tma_load_2d(ring6 + (size_t)u * stage6, &a.tmap_down, ulist[u] * kDExpert, r0,
                        &bars[kBarFull6 + u]);
        }
    }

    // ---------------------------------------------------------- phase 4
    const int Ntot = nU * kDExpert;
    const int nb = (int)(((long long)b * Ntot) / G);
    const int ne = (int)(((long long)(b + 1) * Ntot) / G);
    const int cnt = ne - nb;
    if (!is_producer && warp < a.NS4 && cnt > warp) {
        const uint32_t stage4 = (uint32_t)((gated ? 2 : 1) * rowb);
        unsigned char* slot = ring4 + (size_t)warp * stage4;
        uint64_t* fb = &bars[kBarFull4 + warp];
        const TW* Wg = reinterpret_cast<const TW*>(a.Wg);
        const TW* Wu = reinterpret_cast<const TW*>(a.Wu);
        auto issue = [&](int i) {
            const int q = nb + i;
            const int e = ulist[q >> 6];
            const size_t row = (size_t)e * kDExpert + (q & 63);
            mbar_arrive_expect_tx(fb, stage4);
            if (gated) {
                bulk_g2s(slot, Wg + row * d, (uint32_t)rowb, fb);
                bulk_g2s(slot + rowb, Wu + row * d, (uint32_t)rowb, fb);
            } else {
                bulk_g2s(slot, Wu + row * d, (uint32_t)rowb, fb);
            }
        };
        if (lane == 0) {
            fence_proxy_async_smem();
            issue(warp);
        }
        uint32_t use = 0;
        const TW* gs = reinterpret_cast<const TW*>(slot);
        const TW* us = reinterpret_cast<const TW*>(gated ? slot + rowb : slot);
        for (int i = warp; i < cnt; i += a.NS4) {
            mbar_wait(fb, use & 1u, a.status, lim);
            use++;
            float au[TS], ag[TS];
#pragma unroll
            for (int t = 0; t < TS; t++) au[t] = ag[t] = 0.0f;
            for (int c = lane; c < nchunk; c += 32) {
                float uf[kEl], gf[kEl];
                EL::unpack(reinterpret_cast<const uint4*>(us)[c], uf);
                if (gated) EL::unpack(reinterpret_cast<const uint4*>(gs)[c], gf);
#pragma unroll
                for (int t = 0; t < TS; t++) {
                    if (t < T) {
                        float xf[kEl];
                        EL::unpack(reinterpret_cast<const uint4*>(xs + (size_t)t * d)[c], xf);
#pragma unroll
                        for (int q = 0; q < kEl; q++) au[t] = fmaf(uf[q], xf[q], au[t]);
                        if (gated)
#pragma unroll
                            for (int q = 0; q < kEl; q++) ag[t] = fmaf(gf[q], xf[q], ag[t]);
                    }
                }
            }
            const int q = nb + i;
            const int u = q >> 6, n = q & 63;
            const int e = ulist[u];
#pragma unroll
            for (int t = 0; t < TS; t++) {
                const float su = warp_sum(au[t]);
                const float sg = gated ? warp_sum(ag[t]) : 0.0f;
                if (lane == t && t < T) {
                    const float w = gw[t * E + e];
                    a.h_ws[((size_t)u * T + t) * kDExpert + n] = w == 0.0f ? 0.0f : act_h(a.act, su, sg) * w;
                }
            }
            __syncwarp();
            if (lane == 0 && i + a.NS4 < cnt) {
                fence_proxy_async_smem();
                issue(i + a.NS4);
            }
        }
    }

    grid_barrier(a.bar, a.status, lim);

    // ---------------------------------------------------------- phase 6
    if (is_producer) {
        if (lane == 0) {
            for (int u = kNS6; u < ntiles; u++) {
                const int s = u % kNS6;
                const uint32_t k = (uint32_t)(u / kNS6);
                mbar_wait(&bars[kBarEmpty6 + s], (k - 1u) & 1u, a.status, lim);
                fence_proxy_async_smem();
                mbar_arrive_expect_tx(&bars[kBarFull6 + s], stage6);
                tma_load_2d(ring6 + (size_t)s * stage6, &a.tmap_down, ulist[u] * kDExpert, r0,
                            &bars[kBarFull6 + s]);
            }
        }
        return;
    }
    if (rows == 0) return;

    // consumer warp w accumulates row groups w and w + 8 (4 rows per group,
    // 8 lanes per row, each lane a 16-byte chunk of the 64-wide block)
    constexpr int kChunksPerRow = kDExpert / kEl;       // 8 (bf16) or 16 (fp32)
    constexpr int kChunksPerLane = kChunksPerRow / 8;   // 1 or 2
    const int sub = lane & 7;
    const int rig = lane >> 3;
    float acc[2][TS];
#pragma unroll
    for (int i = 0; i < 2; i++)
#pragma unroll
        for (int t = 0; t < TS; t++) acc[i][t] = 0.0f;
    const int uch = a.uch;
    for (int u = 0; u < ntiles; u++) {
        if (u % uch == 0) {
            named_bar_sync(1, kConsumerWarps * 32);
            const int nu = min(uch, ntiles - u);
            const float4* src = reinterpret_cast<const float4*>(a.h_ws + (size_t)u * T * kDExpert);
            float4* dst = reinterpret_cast<float4*>(hs);
            for (int i = tid; i < nu * T * kDExpert / 4; i += kConsumerWarps * 32) dst[i] = __ldcg(src + i);
            named_bar_sync(1, kConsumerWarps * 32);
        }
        const int s = u % kNS6;
        mbar_wait(&bars[kBarFull6 + s], (uint32_t)(u / kNS6) & 1u, a.status, lim);
        const TW* tile = reinterpret_cast<const TW*>(ring6 + (size_t)s * stage6);
        const float* hu = hs + (size_t)(u % uch) * T * kDExpert;
#pragma unroll
        for (int gi = 0; gi < 2; gi++) {
            const int row = (warp + gi * kConsumerWarps) * 4 + rig;
            if (row < rows) {
#pragma unroll
                for (int cc = 0; cc < kChunksPerLane; cc++) {
                    const int chunk = sub + cc * 8;
                    float wf[kEl];
                    EL::unpack(reinterpret_cast<const uint4*>(tile + (size_t)row * kDExpert)[chunk], wf);
#pragma unroll
                    for (int t = 0; t < TS; t++) {
                        if (t < T) {
                            const float* hv = hu + (size_t)t * kDExpert + chunk * kEl;
#pragma unroll
                            for (int q = 0; q < kEl; q++) acc[gi][t] = fmaf(wf[q], hv[q], acc[gi][t]);
                        }
                    }
                }
            }
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(&bars[kBarEmpty6 + s]);
    }
#pragma unroll
    for (int gi = 0; gi < 2; gi++) {
        const int row = (warp + gi * kConsumerWarps) * 4 + rig;
#pragma unroll
        for (int t = 0; t < TS; t++) {
            float v = acc[gi][t];
            v += __shfl_xor_sync(kFull, v, 1);
            v += __shfl_xor_sync(kFull, v, 2);
            v += __shfl_xor_sync(kFull, v, 4);
            if (sub == 0 && row < rows && t < T) EL::store(a.y, (size_t)t * d + r0 + row, v);
        }
    }
}

// ------------------------------------------------------------------ host
namespace {

size_t align_up(size_t v, size_t a) { return (v + a - 1) / a * a; }

}  // namespace

bool decode_plan(const DecodePlanIn& in, DecodePlan* out) {
    const size_t esz = in.dtype == PP_BF16 ? 2 : 4;
    const int TS = in.TS;
    const int G = in.grid;
    DecodePlan p{};
    p.R6 = (in.d + G - 1) / G;
    if (p.R6 > 2 * kConsumerWarps * 4) return false;  // 64 rows per CTA at most
    size_t off = align_up(kNumBars * 8, 128);
    p.off_x = (uint32_t)off;
    off = align_up(off + (size_t)TS * in.d * esz, 128);
    p.off_gw = (uint32_t)off;
    off = align_up(off + (size_t)TS * in.E * 4, 128);
    p.off_mask = (uint32_t)off;
    off = align_up(off + kMaxExperts * 4, 128);
    p.off_ulist = (uint32_t)off;
    off = align_up(off + kMaxExperts * 4, 128);
    p.off_red = (uint32_t)off;
    off = align_up(off + (size_t)kConsumerWarps * 2 * TS * 4, 128);
    p.uch = (int)std::max<size_t>(1, (16 * 1024) / ((size_t)TS * kDExpert * 4));
    if (p.uch > in.E) p.uch = in.E;
    p.off_h = (uint32_t)off;
    off = align_up(off + (size_t)p.uch * TS * kDExpert * 4, 1024);
    p.off_ring6 = (uint32_t)off;
    off = align_up(off + (size_t)kNS6 * p.R6 * kDExpert * esz, 1024);
    p.off_ring4 = (uint32_t)off;
    const size_t stage4 = (size_t)(in.gated ? 2 : 1) * in.d * esz;
    const size_t budget = in.smem_limit;
    if (off + stage4 > budget) return false;
    int ns4 = (int)std::min<size_t>(kMaxNS4, (budget - off) / stage4);
    // phase 1 reuses the ring for this CTA's router rows
    const int rpc = (in.E + G - 1) / G;
    while ((size_t)ns4 * stage4 < (size_t)rpc * in.d * esz && ns4 < kMaxNS4) ns4++;
    if (off + (size_t)ns4 * stage4 > budget) return false;
    p.NS4 = ns4;
    p.smem = off + (size_t)ns4 * stage4;
    p.threads = kDecThreads;
    *out = p;
    return true;
}

template <typename TW, int TS>
static cudaError_t launch_one(const DecodeArgs& a, const DecodePlan& p, int grid, cudaStream_t st) {
    auto kern = decode_layer_kernel<TW, TS>;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)p.smem);
    if (e != cudaSuccess) return e;
    cudaLaunchConfig_t cfg{};
    cfg.gridDim = dim3(grid);
    cfg.blockDim = dim3(p.threads);
    cfg.dynamicSmemBytes = p.smem;
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeCooperative;
    attr[0].val.cooperative = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kern, a);
}

cudaError_t decode_launch(const DecodeArgs& a, const DecodePlan& p, int dtype, int TS, int grid,
                          cudaStream_t st) {
    if (dtype == PP_BF16) {
        switch (TS) {
            case 1: return launch_one<__nv_bfloat16, 1>(a, p, grid, st);
            case 2: return launch_one<__nv_bfloat16, 2>(a, p, grid, st);
            case 4: return launch_one<__nv_bfloat16, 4>(a, p, grid, st);
            default: return cudaErrorInvalidValue;
        }
    }
    switch (TS) {
        case 1: return launch_one<float, 1>(a, p, grid, st);
        case 2: return launch_one<float, 2>(a, p, grid, st);
        case 4: return launch_one<float, 4>(a, p, grid, st);
        case 8: return launch_one<float, 8>(a, p, grid, st);
        default: return cudaErrorInvalidValue;
    }
}

int decode_max_ts(int dtype) { return dtype == PP_BF16 ? 4 : 8; }

}  // namespace pp
