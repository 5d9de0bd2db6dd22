// MoEfication preprocessing (Sec. 2.2): balanced k-means over the
// intermediate neurons of a dense FFN, and the repacking of its weights into
// contiguous expert blocks (Eq. permuted_weights).
//
// The clustering is an offline host step (it runs once per model, before any
// token is served): the neurons' features are widened into host memory and the
// constrained k-means of Bradley, Bennett and Demiriz (2000) alternates an
// exact equal-size assignment with a centroid update, on the calling thread
// plus a pool of host threads for the distance matrix.  The repacking moves
// the model's weights, which live in HBM: it is a CUDA gather (rows of
// W_gate / W_up, columns of W_down) at copy bandwidth.
#include <algorithm>
#include <atomic>
#include <cmath>
#include <cstring>
#include <limits>
#include <new>
#include <thread>
#include <vector>

#include "pp_common.cuh"
#include "pp_kernels.h"

namespace pp {
namespace {

// ------------------------------------------------------------------ host
float widen_host(const void* base, int dtype, size_t i) {
    if (dtype == PP_F32) return static_cast<const float*>(base)[i];
    const uint32_t u = (uint32_t)static_cast<const uint16_t*>(base)[i] << 16;
    float f;
    std::memcpy(&f, &u, sizeof f);
    return f;
}

// Runs fn(i) for i in [0, n) on up to `threads` host threads (fn must not throw).
template <class Fn>
void parallel_for(int n, int threads, Fn fn) {
    threads = std::max(1, std::min(threads, n));
    if (threads == 1) {
        for (int i = 0; i < n; ++i) fn(i);
        return;
    }
    std::atomic<int> next{0};
    auto body = [&]() {
        for (int i = next.fetch_add(1); i < n; i = next.fetch_add(1)) fn(i);
    };
    std::vector<std::thread> pool;
    pool.reserve(threads - 1);
    try {
        for (int t = 1; t < threads; ++t) pool.emplace_back(body);
    } catch (...) {
        // fewer threads than asked for: the work left runs on those started and here
    }
    body();
    for (auto& th : pool) th.join();
}

// Exact equal-size assignment: n points to k clusters of `cap` points each
// (n == k * cap), minimising sum_i D[i][a[i]].  Min-cost flow by successive
// shortest paths with the points added one at a time: the residual graph is
// contracted onto the clusters (moving point j from cluster h to h2 costs
// D[j][h2] - D[j][h]; the edge h -> h2 keeps the cheapest such j), cluster
// potentials keep every reduced edge cost non-negative, and each point's
// cheapest insertion (directly into a cluster with room, or by a chain of
// moves ending in one) is a dense Dijkstra over the k clusters.  After every
// insertion the assignment of the points added so far is optimal.
class BalancedAssigner {
public:
    BalancedAssigner(const double* D, int n, int k, int cap)
        : D_(D), n_(n), k_(k), cap_(cap), label_(n, -1), members_(k), pot_(k, 0.0),
          w_((size_t)k * k, kInf), wj_((size_t)k * k, -1), dist_(k), parent_(k), done_(k) {
        for (auto& m : members_) m.reserve(cap);
    }

    void run() {
        for (int i = 0; i < n_; ++i) insert(i);
    }
    const std::vector<int>& labels() const { return label_; }

private:
    static constexpr double kInf = std::numeric_limits<double>::infinity();

    double d(int i, int h) const { return D_[(size_t)i * k_ + h]; }

    // edge costs out of cluster h for its current members
    void refresh_row(int h) {
        for (int h2 = 0; h2 < k_; ++h2) {
            double best = kInf;
            int bj = -1;
            if (h2 != h) {
                for (int j : members_[h]) {
                    const double v = d(j, h2) - d(j, h);
                    if (v < best || (v == best && j < bj)) {
                        best = v;
                        bj = j;
                    }
                }
            }
            w_[(size_t)h * k_ + h2] = best;
            wj_[(size_t)h * k_ + h2] = bj;
        }
    }

    void insert(int i) {
        // Dijkstra on reduced costs; dist_ holds true distance - potential
        for (int h = 0; h < k_; ++h) {
            dist_[h] = d(i, h) - pot_[h];
            parent_[h] = -1;
            done_[h] = 0;
        }
        for (int step = 0; step < k_; ++step) {
            int u = -1;
            for (int h = 0; h < k_; ++h)
                if (!done_[h] && (u < 0 || dist_[h] < dist_[u])) u = h;
            done_[u] = 1;
            const double base = dist_[u] + pot_[u];
            const double* wr = &w_[(size_t)u * k_];
            for (int h = 0; h < k_; ++h) {
                if (done_[h] || wr[h] == kInf) continue;
                const double nd = base + wr[h] - pot_[h];
                if (nd < dist_[h]) {
                    dist_[h] = nd;
                    parent_[h] = u;
                }
            }
        }
        // the cheapest cluster with room ends the augmenting path
        int t = -1;
        double tbest = kInf;
        for (int h = 0; h < k_; ++h) {
            if ((int)members_[h].size() >= cap_) continue;
            const double v = dist_[h] + pot_[h];
            if (t < 0 || v < tbest) {
                t = h;
                tbest = v;
            }
        }
        // potentials = true shortest distances (valid for the next search)
        for (int h = 0; h < k_; ++h) pot_[h] += dist_[h];
        // moves along the path, taken from the edges as they were searched
        path_.clear();
        for (int h = t; parent_[h] >= 0; h = parent_[h]) {
            const int from = parent_[h];
            path_.push_back({wj_[(size_t)from * k_ + h], from, h});
        }
        int first = t;
        while (parent_[first] >= 0) first = parent_[first];
        for (const Move& mv : path_) {
            auto& src = members_[mv.from];
            src.erase(std::find(src.begin(), src.end(), mv.j));
            members_[mv.to].push_back(mv.j);
            label_[mv.j] = mv.to;
        }
        members_[first].push_back(i);
        label_[i] = first;
        refresh_row(first);
        for (const Move& mv : path_) refresh_row(mv.to);
    }

    struct Move {
        int j, from, to;
    };

    const double* D_;
    int n_, k_, cap_;
    std::vector<int> label_;
    std::vector<std::vector<int>> members_;
    std::vector<double> pot_, w_;
    std::vector<int> wj_;
    std::vector<double> dist_;
    std::vector<int> parent_;
    std::vector<char> done_;
    std::vector<Move> path_;
};

int host_threads() {
    const unsigned hc = std::thread::hardware_concurrency();
    return (int)std::min(64u, std::max(1u, hc));
}

// D[i][h] = ||F_i||^2 - 2 F_i . C_h + ||C_h||^2 (fp64), 4 clusters per pass
// over a feature row.
void distances(const std::vector<float>& F, const std::vector<double>& fnorm, const std::vector<double>& C,
               int n, int k, int f, std::vector<double>& D, int threads) {
    std::vector<double> cnorm(k);
    for (int h = 0; h < k; ++h) {
        double s = 0.0;
        const double* c = &C[(size_t)h * f];
        for (int x = 0; x < f; ++x) s += c[x] * c[x];
        cnorm[h] = s;
    }
    parallel_for(n, threads, [&](int i) {
        const float* fi = &F[(size_t)i * f];
        int h = 0;
        for (; h + 4 <= k; h += 4) {
            const double* c0 = &C[(size_t)h * f];
            const double* c1 = c0 + f;
            const double* c2 = c1 + f;
            const double* c3 = c2 + f;
            double s0 = 0.0, s1 = 0.0, s2 = 0.0, s3 = 0.0;
            for (int x = 0; x < f; ++x) {
                const double v = fi[x];
                s0 += v * c0[x];
                s1 += v * c1[x];
                s2 += v * c2[x];
                s3 += v * c3[x];
            }
            D[(size_t)i * k + h] = fnorm[i] - 2.0 * s0 + cnorm[h];
            D[(size_t)i * k + h + 1] = fnorm[i] - 2.0 * s1 + cnorm[h + 1];
            D[(size_t)i * k + h + 2] = fnorm[i] - 2.0 * s2 + cnorm[h + 2];
            D[(size_t)i * k + h + 3] = fnorm[i] - 2.0 * s3 + cnorm[h + 3];
        }
        for (; h < k; ++h) {
            const double* c = &C[(size_t)h * f];
            double s = 0.0;
            for (int x = 0; x < f; ++x) s += (double)fi[x] * c[x];
            D[(size_t)i * k + h] = fnorm[i] - 2.0 * s + cnorm[h];
        }
    });
}

// ---------------------------------------------------------------- device
// One CTA: every entry of perm in [0, dff) and none repeated, else the
// status word records PP_ERR_INVALID_ARG.  bitmap: dff bits of shared memory.
__global__ void __launch_bounds__(1024) perm_check_kernel(const int32_t* __restrict__ perm, int dff,
                                                          unsigned* status) {
    extern __shared__ unsigned bitmap[];
    const int words = (dff + 31) >> 5;
    for (int w = threadIdx.x; w < words; w += blockDim.x) bitmap[w] = 0u;
    __syncthreads();
    bool bad = false;
    for (int j = threadIdx.x; j < dff; j += blockDim.x) {
        const int v = perm[j];
        if (v < 0 || v >= dff) {
            bad = true;
            continue;
        }
        const unsigned bit = 1u << (v & 31);
        if (atomicOr(&bitmap[v >> 5], bit) & bit) bad = true;
    }
    if (__syncthreads_or(bad) && threadIdx.x == 0) record_status(status, PP_ERR_INVALID_ARG);
}

// Rows of W_gate / W_up: out[m][j][:] = in[m][perm[j]][:] (a zero row for an
// out-of-range entry, which perm_check_kernel reports).  One row per CTA
// iteration, 16-byte loads and stores; `chunks` = row bytes / 16.
__global__ void __launch_bounds__(256) permute_rows_kernel(const int32_t* __restrict__ perm, const uint4* in0,
                                                           const uint4* in1, uint4* out0, uint4* out1, int dff,
                                                           int nmat, int chunks) {
    const long long rows = (long long)dff * nmat;
    for (long long r = blockIdx.x; r < rows; r += gridDim.x) {
        const int m = (int)(r / dff);
        const int j = (int)(r - (long long)m * dff);
        const int src = perm[j];
        const uint4* in = m == 0 ? in0 : in1;
        uint4* out = (m == 0 ? out0 : out1) + (size_t)j * chunks;
        if (src < 0 || src >= dff) {
            for (int c = threadIdx.x; c < chunks; c += blockDim.x) out[c] = make_uint4(0u, 0u, 0u, 0u);
            continue;
        }
        const uint4* row = in + (size_t)src * chunks;
        for (int c = threadIdx.x; c < chunks; c += blockDim.x) __stcs(out + c, __ldcs(row + c));
    }
}

// Columns of W_down [d][dff]: out[r][j] = in[r][perm[j]].  Each CTA keeps
// perm in shared memory, stages whole rows of W_down there with 16-byte
// loads and writes the gathered row with 16-byte stores.  TE is the 16-bit
// or 32-bit element (bit pattern); VEC = 16 / sizeof(TE).
template <typename TE>
__global__ void __launch_bounds__(512) permute_cols_kernel(const int32_t* __restrict__ perm, const TE* in, TE* out,
                                                           int d, int dff) {
    constexpr int VEC = 16 / (int)sizeof(TE);
    extern __shared__ __align__(16) unsigned char smem[];
    int* perm_s = reinterpret_cast<int*>(smem);
    TE* row_s = reinterpret_cast<TE*>(smem + (size_t)dff * 4);
    for (int j = threadIdx.x; j < dff; j += blockDim.x) {
        const int v = perm[j];
        perm_s[j] = (v >= 0 && v < dff) ? v : -1;
    }
    const int chunks = dff / VEC;
    for (int r = blockIdx.x; r < d; r += gridDim.x) {
        const uint4* src = reinterpret_cast<const uint4*>(in + (size_t)r * dff);
        uint4* srow = reinterpret_cast<uint4*>(row_s);
        __syncthreads();  // perm_s ready; previous row's gather done
        for (int c = threadIdx.x; c < chunks; c += blockDim.x) srow[c] = __ldcs(src + c);
        __syncthreads();
        uint4* dst = reinterpret_cast<uint4*>(out + (size_t)r * dff);
        for (int c = threadIdx.x; c < chunks; c += blockDim.x) {
            union {
                uint4 v;
                TE e[VEC];
            } u;
#pragma unroll
            for (int v = 0; v < VEC; ++v) {
                const int s = perm_s[c * VEC + v];
                u.e[v] = s >= 0 ? row_s[s] : TE(0);
            }
            __stcs(dst + c, u.v);
        }
    }
}

}  // namespace

// ------------------------------------------------------------ interfaces
pp_status moefy_cluster_host(int dtype, const void* Wg, const void* Wu, int dff, int d, int E, const int32_t* init,
                             int max_iter, int32_t* labels, int32_t* perm, int* iters, double* objective) {
    try {
        const int n = dff, cap = dff / E, nsrc = Wg ? 2 : 1;
        const int f = nsrc * d;
        const int threads = host_threads();
        // step 1: features (gate row then up row), exact widening to fp32
        std::vector<float> F((size_t)n * f);
        std::vector<double> fnorm(n);
        parallel_for(n, threads, [&](int i) {
            float* fi = &F[(size_t)i * f];
            for (int s = 0; s < nsrc; ++s) {
                const void* W = (nsrc == 2 && s == 0) ? Wg : Wu;
                for (int x = 0; x < d; ++x) fi[s * d + x] = widen_host(W, dtype, (size_t)i * d + x);
            }
            double q = 0.0;
            for (int x = 0; x < f; ++x) q += (double)fi[x] * fi[x];
            fnorm[i] = q;
        });
        // step 2: balanced k-means from the given neurons' features
        std::vector<double> C((size_t)E * f), D((size_t)n * E);
        for (int h = 0; h < E; ++h)
            for (int x = 0; x < f; ++x) C[(size_t)h * f + x] = F[(size_t)init[h] * f + x];
        std::vector<int> a, prev;
        double obj = 0.0;
        int it = 0;
        while (it < max_iter) {
            ++it;
            distances(F, fnorm, C, n, E, f, D, threads);
            BalancedAssigner as(D.data(), n, E, cap);
            as.run();
            a = as.labels();
            obj = 0.0;
            for (int i = 0; i < n; ++i) obj += D[(size_t)i * E + a[i]];
            if (!prev.empty() && a == prev) break;
            // centroid update: member means
            parallel_for(E, threads, [&](int h) {
                double* c = &C[(size_t)h * f];
                std::fill(c, c + f, 0.0);
                int cnt = 0;
                for (int i = 0; i < n; ++i) {
                    if (a[i] != h) continue;
                    const float* fi = &F[(size_t)i * f];
                    for (int x = 0; x < f; ++x) c[x] += fi[x];
                    ++cnt;
                }
                const double inv = 1.0 / (double)cnt;
                for (int x = 0; x < f; ++x) c[x] *= inv;
            });
            prev = a;
        }
        // step 3: perm = neurons ordered by (cluster, index)
        std::vector<int> fill(E, 0);
        for (int i = 0; i < n; ++i) perm[(size_t)a[i] * cap + fill[a[i]]++] = i;
        if (labels)
            for (int i = 0; i < n; ++i) labels[i] = a[i];
        if (iters) *iters = it;
        if (objective) *objective = obj;
        return PP_OK;
    } catch (...) {
        return PP_ERR_HOST;
    }
}

cudaError_t moefy_permute_launch(int dtype, const int32_t* perm, const void* Wg, const void* Wu, const void* Wd,
                                 void* Wg_out, void* Wu_out, void* Wd_out, int d, int dff, int sms, unsigned* status,
                                 cudaStream_t st) {
    const size_t esz = dtype == PP_BF16 ? 2 : 4;
    perm_check_kernel<<<1, 1024, (size_t)((dff + 31) / 32) * 4, st>>>(perm, dff, status);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    // gate / up rows
    const int nmat = Wg ? 2 : 1;
    const int chunks = (int)((size_t)d * esz / 16);
    const long long rows = (long long)dff * nmat;
    const int grid_rows = (int)std::min<long long>(rows, (long long)sms * 8);
    permute_rows_kernel<<<grid_rows, 256, 0, st>>>(
        perm, static_cast<const uint4*>(Wg ? Wg : Wu), static_cast<const uint4*>(Wu),
        static_cast<uint4*>(Wg ? Wg_out : Wu_out), static_cast<uint4*>(Wu_out), dff, nmat, chunks);
    e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    // down columns
    const size_t smem = (size_t)dff * 4 + (size_t)dff * esz;
    const void* fn = dtype == PP_BF16 ? (const void*)permute_cols_kernel<uint16_t>
                                      : (const void*)permute_cols_kernel<uint32_t>;
    e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    int per_sm = 0;
    e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, fn, 512, smem);
    if (e != cudaSuccess) return e;
    const int grid_cols = std::max(1, std::min(d, sms * std::max(1, per_sm)));
    if (dtype == PP_BF16)
        permute_cols_kernel<uint16_t><<<grid_cols, 512, smem, st>>>(
            perm, static_cast<const uint16_t*>(Wd), static_cast<uint16_t*>(Wd_out), d, dff);
    else
        permute_cols_kernel<uint32_t><<<grid_cols, 512, smem, st>>>(
            perm, static_cast<const uint32_t*>(Wd), static_cast<uint32_t*>(Wd_out), d, dff);
    return cudaGetLastError();
}

}  // namespace pp
