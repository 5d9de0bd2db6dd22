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
