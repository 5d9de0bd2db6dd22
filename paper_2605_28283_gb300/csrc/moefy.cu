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
constexpr uint64_t kPermTimeoutNs = 2000000000ull;  // bounded waits give up after 2 s

// Every entry of perm in [0, dff) and none repeated, else the status word
// records PP_ERR_INVALID_ARG (one CTA of 256 threads; bitmap of dff bits in
// shared memory, dff <= 256 * 64).
PP_DEVINL void perm_check_cta(const int32_t* __restrict__ perm, int dff, unsigned* status) {
    __shared__ unsigned bitmap[kMaxExperts * kDExpert / 32];
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
// out-of-range entry).  Row-gather CTA `cta` of `ncta` takes rows cta,
// cta + ncta, ..., kRowsInFlight of them at a time (every thread loads its
// 16-byte chunk of all of them before storing any), so that enough bytes are
// in flight per CTA; `chunks` = row bytes / 16.
constexpr int kRowsInFlight = 2;
PP_DEVINL void permute_rows_cta(const int32_t* __restrict__ perm, const uint4* in0, const uint4* in1, uint4* out0,
                                uint4* out1, int dff, int nmat, int chunks, int cta, int ncta) {
    const long long rows = (long long)dff * nmat;
    for (long long r0 = cta; r0 < rows; r0 += (long long)ncta * kRowsInFlight) {
        const uint4* src[kRowsInFlight];
        uint4* dst[kRowsInFlight];
#pragma unroll
        for (int k = 0; k < kRowsInFlight; k++) {
            const long long r = r0 + (long long)k * ncta;
            src[k] = nullptr;
            dst[k] = nullptr;
            if (r < rows) {
                const int m = (int)(r / dff);
                const int j = (int)(r - (long long)m * dff);
                const int s = perm[j];
                dst[k] = (m == 0 ? out0 : out1) + (size_t)j * chunks;
                if (s >= 0 && s < dff) src[k] = (m == 0 ? in0 : in1) + (size_t)s * chunks;
            }
        }
        for (int c = threadIdx.x; c < chunks; c += blockDim.x) {
            uint4 v[kRowsInFlight];
#pragma unroll
            for (int k = 0; k < kRowsInFlight; k++) v[k] = src[k] ? __ldcs(src[k] + c) : make_uint4(0u, 0u, 0u, 0u);
#pragma unroll
            for (int k = 0; k < kRowsInFlight; k++)
                if (dst[k]) __stcs(dst[k] + c, v[k]);
        }
    }
}

// The row gather: the last CTA checks perm instead (the gathers do not depend
// on the check, so it runs beside them).
__global__ void __launch_bounds__(256) permute_rows_kernel(const int32_t* __restrict__ perm, const uint4* in0,
                                                           const uint4* in1, uint4* out0, uint4* out1, int dff,
                                                           int nmat, int chunks, unsigned* status) {
    pdl_launch_dependents();  // the column gather (next on the stream) does not read what this grid writes
    if (blockIdx.x == gridDim.x - 1)
        perm_check_cta(perm, dff, status);
    else
        permute_rows_cta(perm, in0, in1, out0, out1, dff, nmat, chunks, (int)blockIdx.x, (int)gridDim.x - 1);
}

// Columns of W_down [d][dff]: out[r][j] = in[r][perm[j]].  Each column CTA keeps
// perm in shared memory (16-bit entries, 0xffff for an out-of-range one) and
// a ring of nbuf whole rows of W_down, filled by 1-D bulk copies: the copy
// of a later row is in flight while the current one is gathered and written
// with 16-byte stores.  TE is the 16-bit or 32-bit element (bit pattern);
// VEC = 16 / sizeof(TE).  Row bytes (dff * sizeof(TE)) are a multiple of 128.
template <typename TE>
__global__ void __launch_bounds__(512) permute_cols_kernel(const int32_t* __restrict__ perm, const TE* in, TE* out,
                                                           int d, int dff, int nbuf, unsigned* status) {
    constexpr int VEC = 16 / (int)sizeof(TE);
    extern __shared__ __align__(128) unsigned char smem[];
    uint64_t* bars = reinterpret_cast<uint64_t*>(smem);  // nbuf <= 4 mbarriers
    uint16_t* perm_s = reinterpret_cast<uint16_t*>(smem + 128);
    TE* ring = reinterpret_cast<TE*>(smem + 128 + (((size_t)dff * 2 + 127) & ~(size_t)127));
    const uint32_t row_bytes = (uint32_t)((size_t)dff * sizeof(TE));
    const int G = gridDim.x;
    if (threadIdx.x == 0) {
        for (int i = 0; i < nbuf; i++) mbar_init(&bars[i], 1);
        fence_mbar_init();
    }
    for (int j = threadIdx.x; j < dff; j += blockDim.x) {
        const int v = perm[j];
        perm_s[j] = (v >= 0 && v < dff) ? (uint16_t)v : (uint16_t)0xffff;
    }
    __syncthreads();
    auto issue = [&](int i) {  // row blockIdx.x + i G -> buffer i % nbuf
        const int r = blockIdx.x + i * G;
        uint64_t* bar = &bars[i % nbuf];
        mbar_arrive_expect_tx(bar, row_bytes);
        bulk_g2s(ring + (size_t)(i % nbuf) * dff, in + (size_t)r * dff, row_bytes, bar);
    };
    if (threadIdx.x == 0)
        for (int i = 0; i < nbuf && blockIdx.x + i * G < d; i++) issue(i);
    const int chunks = dff / VEC;
    for (int i = 0; blockIdx.x + i * G < d; i++) {
        const int r = blockIdx.x + i * G;
        const TE* row_s = ring + (size_t)(i % nbuf) * dff;
        mbar_wait(&bars[i % nbuf], (uint32_t)(i / nbuf) & 1u, status, kPermTimeoutNs);
        uint4* dst = reinterpret_cast<uint4*>(out + (size_t)r * dff);
        for (int c = threadIdx.x; c < chunks; c += blockDim.x) {
            // the chunk's VEC source indices in one shared-memory load
            union {
                uint4 v;
                uint16_t e[8];
            } pi;
            if (VEC == 8) {
                pi.v = reinterpret_cast<const uint4*>(perm_s)[c];
            } else {
                const uint2 h = reinterpret_cast<const uint2*>(perm_s)[c];
                pi.v = make_uint4(h.x, h.y, 0u, 0u);
            }
            union {
                uint4 v;
                TE e[VEC];
            } u;
#pragma unroll
            for (int v = 0; v < VEC; ++v) {
                const uint16_t s = pi.e[v];
                u.e[v] = s != 0xffff ? row_s[s] : TE(0);
            }
            __stcs(dst + c, u.v);
        }
        __syncthreads();  // every thread is done with this buffer
        if (threadIdx.x == 0 && blockIdx.x + (i + nbuf) * G < d) {
            fence_proxy_async_smem();
            issue(i + nbuf);
        }
    }
    // started beside the row gather (programmatic dependent launch): finish
    // only after it, so that work later on the stream sees both
    pdl_wait();
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
    // gate / up rows (plus the permutation check in the last CTA)
    const int nmat = Wg ? 2 : 1;
    const int chunks = (int)((size_t)d * esz / 16);
    const long long rows = (long long)dff * nmat;
    const int grid_rows = (int)std::min<long long>(rows, (long long)sms * 8) + 1;
    permute_rows_kernel<<<grid_rows, 256, 0, st>>>(
        perm, static_cast<const uint4*>(Wg ? Wg : Wu), static_cast<const uint4*>(Wu),
        static_cast<uint4*>(Wg ? Wg_out : Wu_out), static_cast<uint4*>(Wu_out), dff, nmat, chunks, status);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    // down columns: a ring of up to 3 rows per CTA, two CTAs per SM when they fit
    int dev = 0, optin = 0;
    if ((e = cudaGetDevice(&dev)) != cudaSuccess) return e;
    if ((e = cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev)) != cudaSuccess) return e;
    const size_t row_bytes = (size_t)dff * esz;
    const size_t fixed = 128 + (((size_t)dff * 2 + 127) & ~(size_t)127);
    int nbuf = 3;
    while (nbuf > 1 && fixed + nbuf * row_bytes > (size_t)optin / 2 - 1024) nbuf--;
    const size_t smem = fixed + nbuf * row_bytes;
    if (smem > (size_t)optin) return cudaErrorInvalidValue;
    const void* fn = dtype == PP_BF16 ? (const void*)permute_cols_kernel<uint16_t>
                                      : (const void*)permute_cols_kernel<uint32_t>;
    e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    int per_sm = 0;
    e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, fn, 512, smem);
    if (e != cudaSuccess) return e;
    const int grid_cols = std::max(1, std::min(d, sms * std::max(1, per_sm)));
    // launched with programmatic dependent launch: it runs beside the row
    // gather (bound by DRAM) while it is bound by shared memory
    cudaLaunchConfig_t cfg{};
    cfg.gridDim = dim3(grid_cols);
    cfg.blockDim = dim3(512);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    if (dtype == PP_BF16)
        e = cudaLaunchKernelEx(&cfg, permute_cols_kernel<uint16_t>, perm, static_cast<const uint16_t*>(Wd),
                               static_cast<uint16_t*>(Wd_out), d, dff, nbuf, status);
    else
        e = cudaLaunchKernelEx(&cfg, permute_cols_kernel<uint32_t>, perm, static_cast<const uint32_t*>(Wd),
                               static_cast<uint32_t*>(Wd_out), d, dff, nbuf, status);
    if (e != cudaSuccess) return e;
    return cudaGetLastError();
}

}  // namespace pp
