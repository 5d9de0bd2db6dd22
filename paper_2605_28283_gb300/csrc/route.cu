// Router logits for many tokens, stand-alone selection, sparsity statistics
// and the bounded-wait test kernel.
#include "pp_common.cuh"
#include "pp_kernels.h"
#include "pp_select.cuh"

namespace pp {

// ------------------------------------------------------------- selection
// One warp per token: Eq. softmax_prob, the descending order and Eq.
// tau_thresh_activate (see pp_select.cuh).  Writes ids/gates in rank order.
template <int S>
__global__ void __launch_bounds__(256) select_kernel(const float* __restrict__ logits, int T, int E,
                                                     float p, int rule, int gate, int32_t* ids,
                                                     int32_t* counts, float* gates, unsigned* status) {
    const int lane = threadIdx.x & 31;
    const int t = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
    if (t >= T) return;
    const float* row = logits + (size_t)t * E;
    unsigned long long key[S];
    bool finite = true;
    const int k = warp_select<S>([&](int j) { return row[j]; }, E, p, rule, key, &finite);
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
}

// One CTA per token (the latency-oriented counting selection of
// pp_select.cuh, the one the fused decode kernel runs); used for small T.
__global__ void __launch_bounds__(256) select_cta_kernel(const float* __restrict__ logits, int E, float p, int rule,
                                                         int gate, int32_t* ids, int32_t* counts, float* gates,
                                                         unsigned* status) {
    __shared__ __align__(16) CtaSelScratch sc;
    const int t = blockIdx.x;
    bool on;
    int r;
    float g;
    const int k = cta_select_fn([&](int j) { return logits[(size_t)t * E + j]; }, E, p, rule, true, sc, status, &on,
                                &r, &g);
    const int j = threadIdx.x;
    write_selection_row(ids + (size_t)t * E, gates + (size_t)t * E, j, E, k, on, r,
                        on ? (gate == PP_GATE_NONE ? 1.0f : sigmoidf_(g)) : 0.0f);
    if (j == 0) counts[t] = k;
}

constexpr int kCtaSelectMaxT = 64;

cudaError_t select_launch(const float* logits, int T, int E, float p, int rule, int gate,
                          int32_t* ids, int32_t* counts, float* gates, unsigned* status,
                          cudaStream_t st) {
    if (T == 0) return cudaSuccess;
    if (T <= kCtaSelectMaxT) {
        select_cta_kernel<<<T, 256, 0, st>>>(logits, E, p, rule, gate, ids, counts, gates, status);
        return cudaGetLastError();
    }
    const int warps = 8;
    const dim3 grid((T + warps - 1) / warps), block(32 * warps);
    switch (sel_slots_for(E)) {
        case 1: select_kernel<1><<<grid, block, 0, st>>>(logits, T, E, p, rule, gate, ids, counts, gates, status); break;
        case 2: select_kernel<2><<<grid, block, 0, st>>>(logits, T, E, p, rule, gate, ids, counts, gates, status); break;
        case 4: select_kernel<4><<<grid, block, 0, st>>>(logits, T, E, p, rule, gate, ids, counts, gates, status); break;
        default: select_kernel<8><<<grid, block, 0, st>>>(logits, T, E, p, rule, gate, ids, counts, gates, status); break;
    }
    return cudaGetLastError();
}

// ---------------------------------------------------------------- router
// logits[t][j] = sum_i W_r[j][i] * x[t][i] (Eq. routing_logits) for any T,
// fp32 FMA on CUDA cores.  A CTA computes a 64-token x 32-expert tile,
// staging 32-wide k slices of x and W_r in shared memory as fp32.
constexpr int kRT = 64, kRE = 32, kRK = 32;

template <typename TW>
__global__ void __launch_bounds__(256) router_kernel(const TW* __restrict__ x, int T, int d,
                                                     const TW* __restrict__ Wr, int E,
                                                     float* __restrict__ logits) {
    __shared__ float xs[kRK][kRT + 1];
    __shared__ float ws[kRK][kRE + 1];
    const int t0 = blockIdx.x * kRT, j0 = blockIdx.y * kRE;
    const int tid = threadIdx.x;
    const int tj = tid & 31;        // expert within tile
    const int tt = (tid >> 5) * 8;  // 8 tokens per thread
    float acc[8] = {0, 0, 0, 0, 0, 0, 0, 0};
    for (int k0 = 0; k0 < d; k0 += kRK) {
        for (int i = tid; i < kRK * kRT; i += 256) {
            const int kk = i % kRK, r = i / kRK;
            const int t = t0 + r;
            xs[kk][r] = (t < T && k0 + kk < d) ? (float)x[(size_t)t * d + k0 + kk] : 0.0f;
        }
        for (int i = tid; i < kRK * kRE; i += 256) {
            const int kk = i % kRK, r = i / kRK;
            const int j = j0 + r;
            ws[kk][r] = (j < E && k0 + kk < d) ? (float)Wr[(size_t)j * d + k0 + kk] : 0.0f;
        }
        __syncthreads();
#pragma unroll 8
        for (int kk = 0; kk < kRK; kk++) {
            const float w = ws[kk][tj];
#pragma unroll
            for (int q = 0; q < 8; q++) acc[q] = fmaf(w, xs[kk][tt + q], acc[q]);
        }
        __syncthreads();
    }
    const int j = j0 + tj;
    if (j < E)
        for (int q = 0; q < 8; q++) {
            const int t = t0 + tt + q;
            if (t < T) logits[(size_t)t * E + j] = acc[q];
        }
}

cudaError_t router_launch(int dtype, const void* x, int T, int d, const void* Wr, int E,
                          float* logits, cudaStream_t st) {
    if (T == 0) return cudaSuccess;
    const dim3 grid((T + kRT - 1) / kRT, (E + kRE - 1) / kRE), block(256);
    if (dtype == PP_BF16)
        router_kernel<__nv_bfloat16><<<grid, block, 0, st>>>(
            reinterpret_cast<const __nv_bfloat16*>(x), T, d, reinterpret_cast<const __nv_bfloat16*>(Wr), E,
            logits);
    else
        router_kernel<float><<<grid, block, 0, st>>>(reinterpret_cast<const float*>(x), T, d,
                                                     reinterpret_cast<const float*>(Wr), E, logits);
    return cudaGetLastError();
}

// ------------------------------------------------------------ statistics
// acc[0] += sum_t counts[t]; acc[1 + c] += #{t : counts[t] == c}  (s_FFN, Sec. 4.1)
__global__ void stats_kernel(const int32_t* __restrict__ counts, int T, int E, unsigned long long* acc) {
    __shared__ unsigned long long hist[kMaxExperts + 2];
    for (int i = threadIdx.x; i < E + 2; i += blockDim.x) hist[i] = 0ull;
    __syncthreads();
    for (int t = blockIdx.x * blockDim.x + threadIdx.x; t < T; t += gridDim.x * blockDim.x) {
        int c = counts[t];
        c = c < 0 ? 0 : (c > E ? E : c);
        atomicAdd(&hist[0], (unsigned long long)c);
        atomicAdd(&hist[1 + c], 1ull);
    }
    __syncthreads();
    for (int i = threadIdx.x; i < E + 2; i += blockDim.x)
        if (hist[i]) atomicAdd(&acc[i], hist[i]);
}

cudaError_t stats_launch(const int32_t* counts, int T, int E, uint64_t* acc, cudaStream_t st) {
    if (T == 0) return cudaSuccess;
    const int blocks = std::min(152, (T + 255) / 256);
    stats_kernel<<<blocks, 256, 0, st>>>(counts, T, E, reinterpret_cast<unsigned long long*>(acc));
    return cudaGetLastError();
}

// ------------------------------------------------------ router statistics
// Forward values of the router terms of the training objective (Sec. 3.2,
// Eq. entropy_loss and Eq. load_balance_loss; L_gate of Sec. 4.2.3) over a
// batch of logits [T][E].  Pass 1: CTA b takes tokens [64 b, 64 b + 64),
// warp w eight of them, lane l the experts l + 32 s.  Per token the softmax
// is max-shifted in fp32.  part[b] = (column sums of p [E], sum of
// p log(p + eps), sum of sigmoid(g)) over the CTA's tokens, fp32, reduced over
// the warps in a fixed order.  Pass 2 (one CTA of 1024 threads) adds the
// parts pairwise in a fixed tree order and combines the totals in fp64: the
// result is deterministic.  (This GPU's fp64 pipe is narrow, so fp64 is kept
// to the final scalars.)
constexpr int kStatTok = 64;
constexpr int kStatFinal = 1024;

__global__ void __launch_bounds__(256) router_stats_part_kernel(const float* __restrict__ logits, int T, int E,
                                                                float eps, float* __restrict__ part,
                                                                unsigned* status) {
    __shared__ float colw[8][kMaxExperts];
    __shared__ float entw[8], gatew[8];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int S = (E + 31) / 32;
    float col[8] = {0, 0, 0, 0, 0, 0, 0, 0};
    float ent = 0.0f, gsum = 0.0f;
    const int per = kStatTok / 8;
    const int tbeg = blockIdx.x * kStatTok + warp * per, tend = min(T, tbeg + per);
    for (int t = tbeg; t < tend; t++) {
        const float* row = logits + (size_t)t * E;
        float g[8];
        bool fin = true;
        float m = -INFINITY;
#pragma unroll
        for (int s = 0; s < 8; s++) {
            const int j = lane + 32 * s;
            g[s] = (s < S && j < E) ? row[j] : -INFINITY;
            if (s < S && j < E) fin = fin && isfinite(g[s]);
            m = fmaxf(m, g[s]);
        }
        fin = __all_sync(kFull, fin);
        m = warp_max(m);
        float e[8], z = 0.0f;
#pragma unroll
        for (int s = 0; s < 8; s++) {
            e[s] = (s < S && lane + 32 * s < E) ? expf(g[s] - m) : 0.0f;
            z += e[s];
        }
        z = warp_sum(z);
        float te = 0.0f, tg = 0.0f;
#pragma unroll
        for (int s = 0; s < 8; s++) {
            if (s < S && lane + 32 * s < E) {
                const float pj = e[s] / z;
                col[s] += pj;
                te += pj * logf(pj + eps);
                tg += sigmoidf_(g[s]);
            }
        }
        if (!fin) {
            te = __int_as_float(0x7fc00000);  // NaN: the statistics of a batch with a non-finite logit
            if (lane == 0) record_status(status, PP_ERR_NONFINITE);
        }
        ent += te;
        gsum += tg;
    }
#pragma unroll
    for (int s = 0; s < 8; s++)
        if (s < S && lane + 32 * s < E) colw[warp][lane + 32 * s] = col[s];
    ent = warp_sum(ent);
    gsum = warp_sum(gsum);
    if (lane == 0) {
        entw[warp] = ent;
        gatew[warp] = gsum;
    }
    __syncthreads();
    float* out = part + (size_t)blockIdx.x * (E + 2);
    for (int j = threadIdx.x; j < E; j += blockDim.x) {
        float c = 0.0f;
#pragma unroll
        for (int w = 0; w < 8; w++) c += colw[w][j];
        out[j] = c;
    }
    if (threadIdx.x == 0) {
        float a = 0.0f, b = 0.0f;
#pragma unroll
        for (int w = 0; w < 8; w++) {
            a += entw[w];
            b += gatew[w];
        }
        out[E] = a;
        out[E + 1] = b;
    }
}

// Sum of v over the CTA in a fixed tree order (warp shuffles, then warp 0
// over the warp sums); the result is valid in thread 0.
PP_DEVINL float block_sum_fixed(float v, float* red) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = blockDim.x >> 5;
    v = warp_sum(v);
    __syncthreads();  // red may still be read by a previous call
    if (lane == 0) red[warp] = v;
    __syncthreads();
    v = 0.0f;
    if (warp == 0) v = warp_sum(lane < nw ? red[lane] : 0.0f);
    return v;
}

__global__ void __launch_bounds__(kStatFinal) router_stats_final_kernel(const float* __restrict__ part, int nblk,
                                                                        int T, int E, double* __restrict__ out) {
    __shared__ float csum[4][kMaxExperts];
    __shared__ float red[kStatFinal / 32];
    // column sums: four threads per expert, each over a contiguous quarter of
    // the parts, eight loads in flight and a pairwise sum of each eight
    {
        const int j = threadIdx.x >> 2, q = threadIdx.x & 3;
        const int b0 = q * nblk / 4, b1 = (q + 1) * nblk / 4;
        float c = 0.0f;
        if (j < E) {
            int b = b0;
            for (; b + 8 <= b1; b += 8) {
                float v[8];
#pragma unroll
                for (int i = 0; i < 8; i++) v[i] = part[(size_t)(b + i) * (E + 2) + j];
                c += ((v[0] + v[1]) + (v[2] + v[3])) + ((v[4] + v[5]) + (v[6] + v[7]));
            }
            for (; b < b1; b++) c += part[(size_t)b * (E + 2) + j];
            csum[q][j] = c;
        }
    }
    __syncthreads();
    float sq = 0.0f;
    if (threadIdx.x < E) {
        const int j = threadIdx.x;
        const float f = ((csum[0][j] + csum[1][j]) + (csum[2][j] + csum[3][j])) / (float)T;  // (1/B) sum_t p_tj
        sq = f * f;
    }
    float ent = 0.0f, gate = 0.0f;
    for (int b = threadIdx.x; b < nblk; b += blockDim.x) {
        ent += part[(size_t)b * (E + 2) + E];
        gate += part[(size_t)b * (E + 2) + E + 1];
    }
    sq = block_sum_fixed(sq, red);
    ent = block_sum_fixed(ent, red);
    gate = block_sum_fixed(gate, red);
    if (threadIdx.x == 0) {
        out[0] = -(double)ent / (double)T;
        out[1] = (double)E * (double)sq;
        out[2] = (double)gate / ((double)T * (double)E);
    }
}

int router_stats_blocks(int T) { return (T + kStatTok - 1) / kStatTok; }

cudaError_t router_stats_launch(const float* logits, int T, int E, float eps, float* part, double* out,
                                unsigned* status, cudaStream_t st) {
    const int nblk = router_stats_blocks(T);
    router_stats_part_kernel<<<nblk, 256, 0, st>>>(logits, T, E, eps, part, status);
    router_stats_final_kernel<<<1, kStatFinal, 0, st>>>(part, nblk, T, E, out);
    return cudaGetLastError();
}

// ------------------------------------------------------- chained step
// x[t] = RMSNorm(x_prev[t] + y_prev[t]) * gamma, one CTA of 256 threads per
// token: the mean square in fp32 over 16-byte chunks, then the scaled rows
// rounded to the storage type.  The fused decode kernel does the same in its
// prologue; this kernel serves the grouped path and the token slices.
template <typename TW>
__global__ void __launch_bounds__(256) rmsnorm_residual_kernel(const TW* __restrict__ x_prev,
                                                               const TW* __restrict__ y_prev,
                                                               const TW* __restrict__ gamma, float eps, int d,
                                                               TW* __restrict__ x) {
    pdl_wait();  // x_prev / y_prev may be the previous kernel's output
    pdl_launch_dependents();
    using EL = Elem<TW>;
    constexpr int kEl = EL::kPer16B;
    __shared__ float red[8];
    const int t = blockIdx.x, lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int nchunk = d / kEl;
    const uint4* xr = reinterpret_cast<const uint4*>(x_prev + (size_t)t * d);
    const uint4* yr = y_prev ? reinterpret_cast<const uint4*>(y_prev + (size_t)t * d) : nullptr;
    float ss = 0.0f;
    for (int c = threadIdx.x; c < nchunk; c += blockDim.x) {
        float xf[kEl], yf[kEl];
        EL::unpack(xr[c], xf);
        if (yr) EL::unpack(yr[c], yf);
#pragma unroll
        for (int q = 0; q < kEl; q++) {
            const float v = yr ? xf[q] + yf[q] : xf[q];
            ss = fmaf(v, v, ss);
        }
    }
    ss = warp_sum(ss);
    if (lane == 0) red[warp] = ss;
    __syncthreads();
    float tot = 0.0f;
#pragma unroll
    for (int w = 0; w < 8; w++) tot += red[w];
    const float r = rsqrtf(tot / (float)d + eps);
    uint4* xo = reinterpret_cast<uint4*>(x + (size_t)t * d);
    for (int c = threadIdx.x; c < nchunk; c += blockDim.x) {
        float xf[kEl], yf[kEl], gf[kEl];
        EL::unpack(xr[c], xf);
        if (yr) EL::unpack(yr[c], yf);
        if (gamma) EL::unpack(reinterpret_cast<const uint4*>(gamma)[c], gf);
#pragma unroll
        for (int q = 0; q < kEl; q++) xf[q] = (yr ? xf[q] + yf[q] : xf[q]) * r * (gamma ? gf[q] : 1.0f);
        xo[c] = EL::pack(xf);
    }
}

cudaError_t rmsnorm_residual_launch(int dtype, const void* x_prev, const void* y_prev, const void* gamma,
                                    float eps, int T, int d, void* x, cudaStream_t st) {
    if (T == 0) return cudaSuccess;
    cudaLaunchConfig_t cfg{};
    cfg.gridDim = dim3(T);
    cfg.blockDim = dim3(256);
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    if (dtype == PP_BF16) {
        using B = __nv_bfloat16;
        return cudaLaunchKernelEx(&cfg, rmsnorm_residual_kernel<B>, static_cast<const B*>(x_prev),
                                  static_cast<const B*>(y_prev), static_cast<const B*>(gamma), eps, d, static_cast<B*>(x));
    }
    return cudaLaunchKernelEx(&cfg, rmsnorm_residual_kernel<float>, static_cast<const float*>(x_prev),
                              static_cast<const float*>(y_prev), static_cast<const float*>(gamma), eps, d,
                              static_cast<float*>(x));
}

// ------------------------------------------------- bounded wait (test hook)
// Waits for a flag that nothing sets; gives up after timeout_ns and records
// PP_ERR_TIMEOUT.  Exercises the same bounded-wait path the kernels use.
__global__ void wait_timeout_kernel(const unsigned* flag, unsigned* status, long long timeout_ns) {
    if (threadIdx.x != 0) return;
    const uint64_t t0 = globaltimer_ns();
    while (ld_acquire_gpu(flag) == 0u) {
        if ((long long)(globaltimer_ns() - t0) > timeout_ns) {
            record_status(status, PP_ERR_TIMEOUT);
            return;
        }
        __nanosleep(1000);
    }
}

cudaError_t wait_timeout_launch(unsigned* flag, unsigned* status, long long timeout_ns, cudaStream_t st) {
    wait_timeout_kernel<<<1, 32, 0, st>>>(flag, status, timeout_ns);
    return cudaGetLastError();
}

}  // namespace pp
