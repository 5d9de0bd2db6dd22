// Fused decode layer for small token counts (PrunePath Sec. 3.1 end to end).
//
// One cooperative, persistent launch of one CTA (8 warps) per SM does, for
// T <= TS tokens:
//   phase 1  router (Eq. routing_logits): CTA b bulk-loads its rows of W_r
//            and dots them with x (fp32 FMA), publishing each logit as a
//            tagged word (pp_common.cuh);
//   select   every CTA waits for the logits as they arrive, then redundantly
//            selects each token's experts with the CTA-parallel counting
//            selection (Eq. softmax_prob, the descending order, Eq.
//            tau_thresh_activate) and forms U, the union of the tokens'
//            activated experts;
//   phase 4  gate/up (Eq. ffn on the expert blocks): the |U|*64 neurons are
//            split evenly over the grid; each warp bulk-loads the gate and up
//            rows of one neuron into its own shared-memory slot, computes
//            h = act(.) * gate weight (Eq. moe_output) per token and
//            publishes it as a tagged word;
//   phase 6  down projection: CTA b owns R6 rows of W_down and y.  Warp w
//            handles the experts u = w, w+8, ... of U: it streams the
//            [R6 x 64] column block of each with 2-D tensor TMA into its own
//            slots (issued as its phase 4 ends, so that they overlap the h
//            exchange), waits for those experts' h words and accumulates
//            every row of the CTA in registers; one cross-warp reduction in
//            shared memory then writes y once (no atomics: deterministic).
// There is no grid barrier: a CTA waits only for the words it reads.  Each
// launch tags its words with the launch count of the CTA
// (Control.epoch[b], the same in every CTA because every launch runs one CTA
// per SM and each CTA adds 1 to its own count), so words of an earlier
// launch never match.  Only the selected expert blocks are read from HBM.
#include "pp_common.cuh"
#include "pp_kernels.h"
#include "pp_select.cuh"

namespace pp {

constexpr int kWarps = 8;
constexpr int kDecThreads = kWarps * 32;
constexpr int kMaxNS4 = kWarps;
constexpr int kMaxSlots6 = 4;  // phase-6 slots per warp

// barrier indices in the first bytes of shared memory
constexpr int kBarX = 0, kBarR = 1, kBarFull4 = 2, kBarFull6 = kBarFull4 + kMaxNS4,
              kBarH = kBarFull6 + kWarps * kMaxSlots6, kNumBars = kBarH + kWarps;

// Selection given by the caller (pp_sparse_ffn): gates are summed per expert
// so repeated ids behave like repeated terms of the sum.  (Like the other
// paths that the fused layer does not take, kept out of line: the kernel
// runs once per launch and is bound by instruction fetch.)
static __device__ __noinline__ void load_given_selection(const DecodeArgs& a, float* gw, unsigned* mask) {
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

// Selection of every token by the whole CTA, in turn, from the tagged logits
// as they arrive, for the rules other than the cumulative-mass cut (top-k,
// LTE's threshold, p >= 1); CTA 0 publishes it.  Out of line, like
// load_given_selection.
PP_DEVINL void decode_select_cta(const DecodeArgs& a, unsigned tag, float* gw, unsigned* mask, CtaSelScratch& sc) {
    const int tid = threadIdx.x, T = a.T, E = a.E;
    const bool publish = blockIdx.x == 0;
    const bool want_rank = publish && a.sel_ids != nullptr;
    for (int t = 0; t < T; t++) {
        bool on;
        int r;
        float g;
        const unsigned long long* row = a.tlog + (size_t)t * E;
        const int k = cta_select_fn([&](int j) { return wait_tagged(row + j, tag, a.status, a.timeout_ns); }, E, a.p,
                                    a.rule, want_rank, sc, a.status, &on, &r, &g);
        const int j = tid;
        if (j < E) {
            const float gv = on ? (a.gate == PP_GATE_NONE ? 1.0f : sigmoidf_(g)) : 0.0f;
            if (on) {
                gw[t * E + j] = gv;
                mask[j] |= 1u << t;
            }
            if (publish) {
                if (a.sel_ids)
                    write_selection_row(a.sel_ids + (size_t)t * E, a.sel_gates + (size_t)t * E, j, E, k, on, r, gv);
                if (a.sel_logits) a.sel_logits[(size_t)t * E + j] = g;
            }
        }
        if (publish && tid == 0 && a.sel_counts) a.sel_counts[t] = k;
        __syncthreads();  // scratch reuse by the next token
    }
}

// CHAIN: the chained step's prologue (a.chain) is compiled only into its own
// instantiations, so that the plain layer's kernel carries no extra code.
// TL: the timeline instantiation, which also records the global timer at
// the phase boundaries of every CTA into a.tline[CTA][kDecodeStamps] (a
// diagnostic; the plain kernel has no such stores).
template <typename TW, int TS, int RPL, bool CHAIN, bool TL>
__global__ void __launch_bounds__(kDecThreads, 1) decode_layer_kernel(const __grid_constant__ DecodeArgs a) {
    extern __shared__ __align__(1024) unsigned char smem[];
    using EL = Elem<TW>;
    constexpr int kEl = EL::kPer16B;
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
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
    float* red6 = reinterpret_cast<float*>(smem + a.off_red6);
    unsigned char* ring4 = smem + a.off_ring4;
    unsigned char* ring6 = smem + a.off_ring6;
    __shared__ __align__(16) CtaSelScratch sel_sc;
    __shared__ __align__(16) CutShared cut_sc[kWarps];  // one per token group of the cut
    __shared__ int s_nU;
    __shared__ int s_wcount[kWarps];
    __shared__ unsigned s_tag;
    __shared__ int s_k[TS];  // activated experts per token (cumulative-mass cut)
    // timeline stamp i of this CTA (TL instantiation, called by thread 0 only):
    // the global timer at entry, then that plus the SM cycles since entry at
    // kStampMHz (the global timer advances in steps of a few hundred ns)
    uint64_t g0 = 0;
    long long c0 = 0;
    auto stamp = [&](int i) {
        if constexpr (TL)
            a.tline[(size_t)b * kDecodeStamps + i] =
                g0 + (unsigned long long)((clock64() - c0) * 1000ll / kStampMHz);
    };
    if (TL && tid == 0) {
        c0 = clock64();
        g0 = globaltimer_ns();
        stamp(kStEntry);
    }

    if (tid == 0) {
        for (int i = 0; i < kNumBars; i++) mbar_init(&bars[i], 1);
        fence_mbar_init();
    }
    for (int i = tid; i < TS * E; i += kDecThreads) gw[i] = 0.0f;
    for (int i = tid; i < kMaxExperts; i += kDecThreads) mask[i] = 0u;
    if (tid < TS) s_k[tid] = 0;
    __syncthreads();

    // this CTA's router rows of W_r (phase 1): the E rows form blocks of rpc
    // rows, and block j is computed by two CTAs, j and (j + G/2) mod G; they
    // publish the same value, and a reader takes whichever copy arrives first
    // (a CTA that starts late then delays no logit)
    const int rpc = (E + G - 1) / G;
    const int nblk = (E + rpc - 1) / rpc;
    const int blkA = b < nblk ? b : -1;
    const int bB = (b + G / 2) % G;
    const int blkB = bB < nblk && bB != blkA ? bB : -1;
    const int jA = blkA * rpc, jB = blkB * rpc;
    const int nA = a.do_route && blkA >= 0 ? min(E, jA + rpc) - jA : 0;
    const int nB = a.do_route && blkB >= 0 ? min(E, jB + rpc) - jB : 0;
    const int nrows = nA + nB;

    // The router rows are weights: load them before waiting for the
    // preceding grid (with programmatic dependent launch this overlaps the
    // previous layer's tail).  x and the workspace may be that grid's output
    // or scratch, so they are touched only after the wait.
    if (tid == 0 && nrows > 0) {
        const TW* wr = reinterpret_cast<const TW*>(a.Wr);
        mbar_arrive_expect_tx(&bars[kBarR], (uint32_t)(nrows * rowb));
        if (nA > 0) bulk_g2s(ring4, wr + (size_t)jA * d, (uint32_t)(nA * rowb), &bars[kBarR]);
        if (nB > 0) bulk_g2s(ring4 + (size_t)nA * rowb, wr + (size_t)jB * d, (uint32_t)(nB * rowb), &bars[kBarR]);
    }
    pdl_wait();
    pdl_launch_dependents();
    if (TL && tid == 0) stamp(kStReleased);
    TW* chain_y = reinterpret_cast<TW*>(ring4 + a.off_chain);
    TW* chain_g = chain_y + (size_t)TS * d;
    if (tid == 0) {
        const uint32_t bytes = (uint32_t)(T * rowb);  // x -> shared memory (all T rows are contiguous)
        const bool cy = CHAIN && a.y_prev, cg = CHAIN && a.gamma;
        mbar_arrive_expect_tx(&bars[kBarX], bytes + (cy ? bytes : 0u) + (cg ? (uint32_t)rowb : 0u));
        bulk_g2s(xs, a.x, bytes, &bars[kBarX]);
        if (cy) bulk_g2s(chain_y, a.y_prev, bytes, &bars[kBarX]);
        if (cg) bulk_g2s(chain_g, a.gamma, (uint32_t)rowb, &bars[kBarX]);
        // this launch's tag: the CTA's launch count + 1 (its own word, last
        // written by this CTA in the previous launch, which has completed)
        const unsigned ep = a.epochs[b];
        a.epochs[b] = ep + 1u;
        s_tag = ep + 1u;
    }
    // every CTA waits for its copy of x here, so no bulk copy is ever still
    // in flight when a CTA that has no work left exits
    mbar_wait(&bars[kBarX], 0, a.status, lim);
    __syncthreads();
    const unsigned tag = s_tag;
    if (TL && tid == 0) stamp(kStX);

    // chained step: the layer input is RMSNorm(x_prev + y_prev) * gamma, formed
    // in place in shared memory by every CTA (CTA 0 also stores it)
    if (CHAIN) {
        for (int t = 0; t < T; t++) {
            TW* xr = xs + (size_t)t * d;
            const TW* yr = chain_y + (size_t)t * d;
            float ss = 0.0f;
            for (int c = tid; c < nchunk; c += kDecThreads) {
                float xf[kEl], yf[kEl];
                EL::unpack(reinterpret_cast<const uint4*>(xr)[c], xf);
                if (a.y_prev) EL::unpack(reinterpret_cast<const uint4*>(yr)[c], yf);
#pragma unroll
                for (int q = 0; q < kEl; q++) {
                    const float v = a.y_prev ? xf[q] + yf[q] : xf[q];
                    ss = fmaf(v, v, ss);
                }
            }
            ss = warp_sum(ss);
            if (lane == 0) red[warp] = ss;
            __syncthreads();
            float tot = 0.0f;
#pragma unroll
            for (int w = 0; w < kWarps; w++) tot += red[w];
            const float r = rsqrtf(tot / (float)d + a.eps);
            for (int c = tid; c < nchunk; c += kDecThreads) {
                float xf[kEl], yf[kEl], gf[kEl];
                EL::unpack(reinterpret_cast<const uint4*>(xr)[c], xf);
                if (a.y_prev) EL::unpack(reinterpret_cast<const uint4*>(yr)[c], yf);
                if (a.gamma) EL::unpack(reinterpret_cast<const uint4*>(chain_g)[c], gf);
#pragma unroll
                for (int q = 0; q < kEl; q++) {
                    const float v = a.y_prev ? xf[q] + yf[q] : xf[q];
                    xf[q] = v * r * (a.gamma ? gf[q] : 1.0f);
                }
                const uint4 packed = EL::pack(xf);
                reinterpret_cast<uint4*>(xr)[c] = packed;
                if (b == 0) reinterpret_cast<uint4*>(static_cast<TW*>(a.x_out) + (size_t)t * d)[c] = packed;
            }
            __syncthreads();  // red is reused by the next token
        }
    }

    // gate/up rows of global neuron q (neuron q & 63 of the expert at
    // position q >> 6 of U) -> phase-4 ring slot `slot`
    const uint32_t stage4 = (uint32_t)((gated ? 2 : 1) * rowb);
    const TW* Wg = reinterpret_cast<const TW*>(a.Wg);
    const TW* Wu = reinterpret_cast<const TW*>(a.Wu);
    auto issue_row = [&](int q, int slot) {
        const size_t row = (size_t)ulist[q >> 6] * kDExpert + (q & 63);
        unsigned char* dst = ring4 + (size_t)slot * stage4;
        uint64_t* fb = &bars[kBarFull4 + slot];
        mbar_arrive_expect_tx(fb, stage4);
        if (gated) {
            bulk_g2s(dst, Wg + row * d, (uint32_t)rowb, fb);
            bulk_g2s(dst + rowb, Wu + row * d, (uint32_t)rowb, fb);
        } else {
            bulk_g2s(dst, Wu + row * d, (uint32_t)rowb, fb);
        }
    };
    const bool mass_cut = (a.rule == PP_SEL_MIN_PREFIX || a.rule == PP_SEL_PAPER) && a.p < 1.0f;

    // ---------------------------------------------------------- phase 1
    if (a.do_route) {
        if (nrows > 0) {
            mbar_wait(&bars[kBarR], 0, a.status, lim);
            const TW* rows_s = reinterpret_cast<const TW*>(ring4);
            for (int r0 = 0; r0 < nrows; r0 += 2) {
                float acc[2][TS];
#pragma unroll
                for (int i = 0; i < 2; i++)
#pragma unroll
                    for (int t = 0; t < TS; t++) acc[i][t] = 0.0f;
                for (int c = tid; c < nchunk; c += kDecThreads) {
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
                __syncthreads();
                if (tid < 2 * TS) {
                    const int i = tid / TS, t = tid % TS;
                    if (r0 + i < nrows && t < T) {
                        float v = 0.0f;
                        for (int w = 0; w < kWarps; w++) v += red[(w * 2 + i) * TS + t];
                        const int ri = r0 + i;
                        st_tagged(a.tlog + (size_t)t * E + (ri < nA ? jA + ri : jB + ri - nA), tag, v);
                    }
                }
                __syncthreads();
            }
        }
        if (TL && tid == 0) stamp(kStRouter);
        const bool publish = b == 0;
        if (mass_cut) {
            // cumulative-mass cut of every token: the tokens are cut side by
            // side by groups of nt threads (the smallest of 32, 64, 128, 256
            // that holds E experts; up to TS groups, each with its own named
            // barrier); thread j of a group waits for logit j of its token,
            // and every activated expert is recorded by the thread that
            // decides it.  Candidate scratch in the phase-6 ring, idle until
            // phase 6 (the phase-4 ring takes gate/up rows requested during
            // the count).
            const int nt = E <= 32 ? 32 : E <= 64 ? 64 : E <= 128 ? 128 : kDecThreads;
            const int ng = min(TS, kDecThreads / nt);
            const int grp = tid / nt, gj = tid % nt;
            const int bid = nt == kDecThreads ? 0 : 1 + grp;
            WarpCand* cand = reinterpret_cast<WarpCand*>(ring6) + (size_t)grp * nt;
            for (int t0 = 0; t0 < T; t0 += ng) {
                const int t = t0 + grp;
                if (grp >= ng || t >= T) continue;
                const float g = gj < E ? wait_tagged(a.tlog + (size_t)t * E + gj, tag, a.status, lim) : -INFINITY;
                if (TL) {  // timeline only: the moment every logit has arrived
                    group_bar(bid, nt);
                    if (tid == 0 && t == 0) stamp(kStLogits);
                }
                const int k = group_mass_cut(g, E, a.p, a.rule, cut_sc[grp], cand, a.status, bid, nt, [&](int r, int e, float ge) {
                    if (TS == 1) {
                        ulist[r] = e;  // one token: U is its activated set, in rank order
                        // this CTA's neurons q = b + G i of rank r (q in
                        // [64 r, 64 r + 64)) are requested right away, into
                        // slot i, by the thread that activated the expert
                        if (a.do_ffn) {
                            const int lo = r * kDExpert;
                            int q = b, i = 0;
                            while (q < lo) {
                                q += G;
                                i++;
                            }
                            for (; q < lo + kDExpert && i < a.NS4; q += G, i++) {
                                fence_proxy_async_smem();
                                issue_row(q, i);
                            }
                        }
                    } else {
                        atomicOr(&mask[e], 1u << t);  // tokens of other groups at the same time
                    }
                    const float gv = a.gate == PP_GATE_NONE ? 1.0f : sigmoidf_(ge);
                    gw[t * E + e] = gv;
                    if (publish && a.sel_ids) {
                        a.sel_ids[(size_t)t * E + r] = e;
                        a.sel_gates[(size_t)t * E + r] = gv;
                    }
                }, [&] {
                    if (TL && tid == 0 && t == 0) stamp(kStCand);
                });
                if (gj == 0) s_k[t] = k;
                if (publish) {
                    if (a.sel_ids)
                        for (int r = k + gj; r < E; r += nt) {
                            a.sel_ids[(size_t)t * E + r] = -1;
                            a.sel_gates[(size_t)t * E + r] = 0.0f;
                        }
                    if (a.sel_logits && gj < E) a.sel_logits[(size_t)t * E + gj] = g;
                    if (gj == 0 && a.sel_counts) a.sel_counts[t] = k;
                }
            }
            if (TL && tid == 0) stamp(kStCut);
            // the candidate lists in the ring are dead: order their generic
            // accesses before the bulk copies into the ring
            fence_proxy_async_smem();
        } else {
            decode_select_cta(a, tag, gw, mask, sel_sc);
        }
    } else {
        load_given_selection(a, gw, mask);
    }
    __syncthreads();
    if (TL && tid == 0) stamp(kStSelected);
    if (!a.do_ffn) return;

    // union U of the tokens' activated experts, ascending expert index
    // (already formed, in rank order, by the one-token cut)
    if (!(a.do_route && mass_cut && TS == 1)) {
        const int e = tid;
        const bool on = e < E && mask[e] != 0u;
        const unsigned bal = __ballot_sync(kFull, on);
        if (lane == 0) s_wcount[warp] = __popc(bal);
        __syncthreads();
        if (tid == 0) {
            int acc = 0;
            for (int w = 0; w < kWarps; w++) {
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
    const int nU = a.do_route && mass_cut && TS == 1 ? s_k[0] : s_nU;
    if (TL && tid == 0) stamp(kStUnion);

    // phase-6 geometry: CTA b owns rows [r0, r0 + rows) of W_down and y;
    // warp w handles experts u = w + 8 i of U (i < nt_w)
    const int R6 = a.R6;
    const int r0 = b * R6;
    const int rows = max(0, min(R6, d - r0));
    const uint32_t stage6 = (uint32_t)(R6 * kDExpert * sizeof(TW));
    const int ntiles = rows > 0 ? nU : 0;
    const int nt_w = ntiles > warp ? (ntiles - warp + kWarps - 1) / kWarps : 0;
    const int ded6 = a.ded6, slots6 = a.slots6;
    // a warp's first ded6 slots are its own part of the phase-6 ring; the
    // others are carved from the phase-4 ring, free once this CTA's phase 4
    // is done
    auto slot6 = [&](int s) -> unsigned char* {
        return s < ded6 ? ring6 + (size_t)(warp * ded6 + s) * stage6
                        : ring4 + (size_t)(warp * (slots6 - ded6) + (s - ded6)) * stage6;
    };
    auto issue6 = [&](int i) {
        const int s = i % slots6;
        uint64_t* fb = &bars[kBarFull6 + warp * kMaxSlots6 + s];
        mbar_arrive_expect_tx(fb, stage6);
        tma_load_2d(slot6(s), &a.tmap_down, ulist[warp + kWarps * i] * kDExpert, r0, fb);
    };

    // ---------------------------------------------------------- phase 4
    // neurons are dealt round robin: neuron i of this CTA is global neuron
    // q = b + G i (neuron q & 63 of the expert at position q >> 6 of U)
    const int Ntot = nU * kDExpert;
    const int cnt = Ntot > b ? (Ntot - 1 - b) / G + 1 : 0;
    // the one-token cut has already requested neurons i < min(cnt, NS4)
    const bool early = a.do_route && mass_cut && TS == 1;
    auto issue4 = [&](int i, int slot) { issue_row(b + G * i, slot); };
    // dot products of one neuron's gate/up rows (in `slot`) with x over the
    // 16-byte chunks [c0, c1), per token
    auto neuron_dots = [&](int slot, int c0, int c1, float (&au)[TS], float (&ag)[TS]) {
        const unsigned char* base = ring4 + (size_t)slot * stage4;
        const TW* gs = reinterpret_cast<const TW*>(base);
        const TW* us = reinterpret_cast<const TW*>(gated ? base + rowb : base);
#pragma unroll
        for (int t = 0; t < TS; t++) au[t] = ag[t] = 0.0f;
        for (int c = c0 + lane; c < c1; c += 32) {
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
#pragma unroll
        for (int t = 0; t < TS; t++) {
            au[t] = warp_sum(au[t]);
            ag[t] = gated ? warp_sum(ag[t]) : 0.0f;
        }
    };
    auto store_h = [&](int i, int t, float su, float sg) {
        const int q = b + G * i;
        const int u = q >> 6, n = q & 63;
        const float w = gw[t * E + ulist[u]];
        st_tagged(a.th + ((size_t)u * T + t) * kDExpert + n, tag, w == 0.0f ? 0.0f : act_h(a.act, su, sg) * w);
    };
    // Few neurons (cnt <= NS4): all loads at once, neuron i -> slot i, each
    // neuron split into S column slices worked on by S warps.  Many neurons:
    // warp w streams neurons w, w + NS4, ... through slot w.
    const bool few = cnt > 0 && cnt <= a.NS4;
    const int S = cnt == 1 ? 8 : cnt == 2 ? 4 : cnt <= 4 ? 2 : 1;
    if (few && !early && tid == 0) {
        fence_proxy_async_smem();
        for (int i = 0; i < cnt; i++) issue4(i, i);
    }
    if (!few && !early && warp < a.NS4 && cnt > warp && lane == 0) {
        fence_proxy_async_smem();
        issue4(warp, warp);
    }
    if (TL && tid == 0) stamp(kStIssued4);
    if (few) {
        if (warp < cnt * S) {
            const int i = warp / S, sl = warp % S;
            const int cs = (nchunk + S - 1) / S;
            mbar_wait(&bars[kBarFull4 + i], 0, a.status, lim);
            if (TL && tid == 0) stamp(kStLanded4);
            float au[TS], ag[TS];
            neuron_dots(i, sl * cs, min(nchunk, (sl + 1) * cs), au, ag);
#pragma unroll
            for (int t = 0; t < TS; t++) {
                if (lane == t && t < T) {
                    if (S == 1) {
                        store_h(i, t, au[t], ag[t]);
                    } else {
                        red[(warp * 2 + 0) * TS + t] = au[t];
                        red[(warp * 2 + 1) * TS + t] = ag[t];
                    }
                }
            }
        }
        if (S > 1) {
            __syncthreads();
            if (tid < cnt * T) {
                const int i = tid / T, t = tid % T;
                float su = 0.0f, sg = 0.0f;
                for (int sl = 0; sl < S; sl++) {
                    su += red[((i * S + sl) * 2 + 0) * TS + t];
                    sg += red[((i * S + sl) * 2 + 1) * TS + t];
                }
                store_h(i, t, su, sg);
            }
        }
    } else if (cnt > 0 && warp < a.NS4 && cnt > warp) {
        uint32_t use = 0;
        for (int i = warp; i < cnt; i += a.NS4) {
            mbar_wait(&bars[kBarFull4 + warp], use & 1u, a.status, lim);
            use++;
            float au[TS], ag[TS];
            neuron_dots(warp, 0, nchunk, au, ag);
#pragma unroll
            for (int t = 0; t < TS; t++)
                if (lane == t && t < T) store_h(i, t, au[t], ag[t]);
            __syncwarp();
            if (lane == 0 && i + a.NS4 < cnt) {
                fence_proxy_async_smem();
                issue4(i + a.NS4, warp);
            }
        }
    }

    // W_down tiles of phase 6: issued only now, so that across the grid the
    // gate/up bytes that phase 4 waits for are not queued behind W_down bytes
    // (the h exchange that phase 6 waits for anyway covers their latency)
    __syncwarp();
    if (lane == 0) {
        fence_proxy_async_smem();
        for (int i = 0; i < min(nt_w, ded6); i++) issue6(i);
    }
    // this CTA's phase-4 slots are free again (extra phase-6 slots below)
    __syncthreads();
    if (TL && tid == 0) stamp(kStPhase4);

    // ---------------------------------------------------------- phase 6
    if (rows == 0) {
        if (TL && tid == 0) stamp(kStEnd);
        return;
    }
    if (lane == 0) {
        fence_proxy_async_smem();
        for (int i = ded6; i < min(nt_w, slots6); i++) issue6(i);
    }

    // lane: chunk column c of the 64-wide block (8 elements; fp32 uses two
    // 4-element chunks c and c + 8) and rows rig + 4 j
    constexpr int kCPL = kDExpert / kEl / 8;  // 16-byte chunks per lane per row: 1 (bf16) or 2 (fp32)
    const int c = lane & 7, rig = lane >> 3;
    float acc[RPL][TS];
#pragma unroll
    for (int j = 0; j < RPL; j++)
#pragma unroll
        for (int t = 0; t < TS; t++) acc[j][t] = 0.0f;
    // h of this warp's experts, hch experts at a time: bulk copies of their
    // tagged words (written by the CTAs that own the experts' neurons) into
    // the warp's part of the h area, repeated until every word carries this
    // launch's tag
    const int hch = a.hch;
    const int hwords = T * kDExpert;  // h words of one expert slot
    unsigned long long* hs_w =
        reinterpret_cast<unsigned long long*>(ring4 + (size_t)kWarps * (slots6 - ded6) * stage6) +
        (size_t)warp * hch * hwords;
    uint64_t* hbar = &bars[kBarH + warp];
    uint32_t hphase = 0;
    for (int i = 0; i < nt_w; i++) {
        const int u = warp + kWarps * i;
        if (i % hch == 0) {
            const int nc = min(hch, nt_w - i);
            const int npairs = nc * hwords / 2;
            uint64_t t0 = 0;
            bool ready;
            do {
                __syncwarp();  // earlier reads of the area are done
                if (lane == 0) {
                    fence_proxy_async_smem();
                    mbar_arrive_expect_tx(hbar, (uint32_t)(nc * hwords * 8));
                    for (int ti = 0; ti < nc; ti++)
                        bulk_g2s(hs_w + (size_t)ti * hwords, a.th + (size_t)(u + kWarps * ti) * hwords,
                                 (uint32_t)(hwords * 8), hbar);
                }
                mbar_wait(hbar, hphase & 1u, a.status, lim);
                hphase++;
                ready = true;
                for (int q = lane; q < npairs; q += 32) {
                    const ulonglong2 w2 = reinterpret_cast<const ulonglong2*>(hs_w)[q];
                    ready = ready && word_tag(w2.x) == tag && word_tag(w2.y) == tag;
                }
                ready = __all_sync(kFull, ready);
                if (!ready) __nanosleep(kPollBackoffNs);
            } while (!ready && !__shfl_sync(kFull, (int)poll_give_up(t0, a.status, lim), 0));
            if (TL && i == 0 && tid == 0) stamp(kStFirstH);
        }
        const unsigned long long* hu = hs_w + (size_t)(i % hch) * hwords;
        float hv[TS][kCPL * kEl];
#pragma unroll
        for (int t = 0; t < TS; t++)
            if (t < T)
#pragma unroll
                for (int cc = 0; cc < kCPL; cc++) {
                    const ulonglong2* h2 =
                        reinterpret_cast<const ulonglong2*>(hu + (size_t)t * kDExpert + (c + 8 * cc) * kEl);
#pragma unroll
                    for (int q2 = 0; q2 < kEl / 2; q2++) {
                        const ulonglong2 v = h2[q2];
                        hv[t][cc * kEl + q2 * 2 + 0] = word_value(v.x);
                        hv[t][cc * kEl + q2 * 2 + 1] = word_value(v.y);
                    }
                }
        const int s = i % slots6;
        mbar_wait(&bars[kBarFull6 + warp * kMaxSlots6 + s], (uint32_t)(i / slots6) & 1u, a.status, lim);
        const TW* tile = reinterpret_cast<const TW*>(slot6(s));
#pragma unroll
        for (int j = 0; j < RPL; j++) {
            const int row = rig + 4 * j;
            if (row < rows) {
#pragma unroll
                for (int cc = 0; cc < kCPL; cc++) {
                    float wf[kEl];
                    EL::unpack(reinterpret_cast<const uint4*>(tile + (size_t)row * kDExpert)[c + 8 * cc], wf);
#pragma unroll
                    for (int t = 0; t < TS; t++)
                        if (t < T)
#pragma unroll
                            for (int q = 0; q < kEl; q++) acc[j][t] = fmaf(wf[q], hv[t][cc * kEl + q], acc[j][t]);
                }
            }
        }
        __syncwarp();
        if (lane == 0 && i + slots6 < nt_w) {
            fence_proxy_async_smem();
            issue6(i + slots6);
        }
    }
    if (TL && tid == 0) stamp(kStPhase6);
    // reduce over the 8 lanes of a row, then over the warps (fixed order)
#pragma unroll
    for (int j = 0; j < RPL; j++) {
        const int row = rig + 4 * j;
#pragma unroll
        for (int t = 0; t < TS; t++) {
            float v = acc[j][t];
            v += __shfl_xor_sync(kFull, v, 1);
            v += __shfl_xor_sync(kFull, v, 2);
            v += __shfl_xor_sync(kFull, v, 4);
            if (c == 0 && row < rows && t < T) red6[(warp * R6 + row) * TS + t] = v;
        }
    }
    __syncthreads();
    for (int o = tid; o < rows * T; o += kDecThreads) {
        const int row = o / T, t = o % T;
        float v = 0.0f;
        for (int w = 0; w < kWarps; w++)
            if (w < ntiles) v += red6[(w * R6 + row) * TS + t];
        EL::store(a.y, (size_t)t * d + r0 + row, v);
    }
    if (TL && tid == 0) stamp(kStEnd);
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
    if (p.R6 > 64) return false;  // 64 rows per CTA at most (16 per lane)
    p.RPL = (p.R6 + 3) / 4 <= 8 ? 8 : 16;
    const size_t stage6 = (size_t)p.R6 * kDExpert * esz;
    const size_t stage4 = (size_t)(in.gated ? 2 : 1) * in.d * esz;
    const int rpc = (in.E + G - 1) / G;
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
    off = align_up(off + (size_t)kWarps * 2 * TS * 4, 128);
    p.off_red6 = (uint32_t)off;
    off = align_up(off + (size_t)kWarps * p.R6 * TS * 4, 1024);
    const size_t budget = in.smem_limit;
    // dedicated phase-6 slots: 2 per warp when they fit comfortably, else 1
    p.ded6 = (off + 2 * kWarps * stage6 + 2 * stage4 <= budget) ? 2 : 1;
    p.off_ring6 = (uint32_t)off;  // also the cumulative-mass cut's candidate scratch before phase 6
    off = align_up(off + std::max((size_t)p.ded6 * kWarps * stage6, (size_t)kWarps * 32 * sizeof(WarpCand)), 1024);
    p.off_ring4 = (uint32_t)off;
    if (off + stage4 > budget) return false;
    const size_t avail = budget - off;
    // the ring also stages the router rows and, for a chained step, y_prev
    // [TS][d] and gamma [d] (all read before phase 4 uses the ring)
    p.off_chain = (uint32_t)align_up((size_t)2 * rpc * in.d * esz, 128);  // up to two blocks of router rows
    const size_t chain_end =
        in.chain ? (size_t)p.off_chain + align_up((size_t)(TS + 1) * in.d * esz, 128) : (size_t)2 * rpc * in.d * esz;
    const int ns4 = (int)std::min<size_t>(kMaxNS4, avail / stage4);
    // the ring also holds this CTA's router rows (phase 1) and, once phase 4
    // is done, the extra phase-6 slots plus at least one expert's h per warp
    const size_t hper = (size_t)TS * kDExpert * 8;  // tagged h words of one expert
    size_t ring4 = 0;
    int ext = kMaxSlots6 - p.ded6;
    for (; ext >= 0; ext--) {
        ring4 = std::max({(size_t)ns4 * stage4, chain_end,
                          (size_t)ext * kWarps * stage6 + kWarps * hper});
        if (ring4 <= avail) break;
    }
    if (ext < 0) return false;
    p.slots6 = p.ded6 + ext;
    const size_t harea = ring4 - (size_t)ext * kWarps * stage6;
    p.hch = (int)std::min<size_t>((kMaxExperts + kWarps - 1) / kWarps, harea / (kWarps * hper));
    p.NS4 = ns4;
    p.smem = off + ring4;
    p.threads = kDecThreads;
    *out = p;
    return true;
}

template <typename TW, int TS, int RPL, bool TL = false>
static cudaError_t launch_one(const DecodeArgs& a, const DecodePlan& p, int grid, cudaStream_t st) {
    auto kern = TL ? decode_layer_kernel<TW, TS, RPL, false, true>
                   : (a.chain ? decode_layer_kernel<TW, TS, RPL, true, false> : decode_layer_kernel<TW, TS, RPL, false, false>);
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)p.smem);
    if (e != cudaSuccess) return e;
    cudaLaunchConfig_t cfg{};
    cfg.gridDim = dim3(grid);
    cfg.blockDim = dim3(p.threads);
    cfg.dynamicSmemBytes = p.smem;
    cfg.stream = st;
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeCooperative;
    attr[0].val.cooperative = 1;
    attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[1].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 2;
    e = cudaLaunchKernelEx(&cfg, kern, a);
    if (e == cudaErrorNotSupported || e == cudaErrorInvalidValue) {
        (void)cudaGetLastError();  // this runtime cannot combine the two attributes
        cfg.numAttrs = 1;
        e = cudaLaunchKernelEx(&cfg, kern, a);
    }
    return e;
}

template <typename TW, int TS>
static cudaError_t launch_rpl(const DecodeArgs& a, const DecodePlan& p, int grid, cudaStream_t st) {
    return p.RPL == 8 ? launch_one<TW, TS, 8>(a, p, grid, st) : launch_one<TW, TS, 16>(a, p, grid, st);
}

cudaError_t decode_launch(const DecodeArgs& a, const DecodePlan& p, int dtype, int TS, int grid,
                          cudaStream_t st) {
    if (grid < 1 || grid > kMaxGrid) return cudaErrorInvalidValue;  // one launch count per CTA
    if (a.tline) {  // the timeline instantiation exists for one bf16 token of a plain layer only
        if (dtype != PP_BF16 || TS != 1 || a.chain) return cudaErrorInvalidValue;
        return p.RPL == 8 ? launch_one<__nv_bfloat16, 1, 8, true>(a, p, grid, st)
                          : launch_one<__nv_bfloat16, 1, 16, true>(a, p, grid, st);
    }
    if (dtype == PP_BF16) {
        switch (TS) {
            case 1: return launch_rpl<__nv_bfloat16, 1>(a, p, grid, st);
            case 2: return launch_rpl<__nv_bfloat16, 2>(a, p, grid, st);
            case 4: return launch_rpl<__nv_bfloat16, 4>(a, p, grid, st);
            default: return cudaErrorInvalidValue;
        }
    }
    switch (TS) {
        case 1: return launch_rpl<float, 1>(a, p, grid, st);
        case 2: return launch_rpl<float, 2>(a, p, grid, st);
        case 4: return launch_rpl<float, 4>(a, p, grid, st);
        case 8: return launch_rpl<float, 8>(a, p, grid, st);
        default: return cudaErrorInvalidValue;
    }
}

int decode_max_ts(int dtype) { return dtype == PP_BF16 ? 4 : 8; }

}  // namespace pp
