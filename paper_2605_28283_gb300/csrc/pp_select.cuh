// Warp-level cumulative-mass expert selection for one token (PrunePath
// Sec. 3.1: Eq. softmax_prob, the descending order pi, Eq.
// tau_thresh_activate).
//
// One warp holds the token's E <= 32*S logits as 64-bit rank keys, S per
// lane, sorts them with a register bitonic network (in-lane exchanges for
// strides < S, shuffles otherwise), then forms the max-shifted fp32
// exponentials in rank order and their inclusive prefix sums in fp64.  The
// cut compares each prefix with p * Z in fp64.  After the sort lane l holds
// ranks l*S .. l*S+S-1 in key[0..S-1].  The same order serves the top-k rule
// (Sec. 4.3) and LTE's threshold rule (Eq. lte_hard_set).
#pragma once

#include "pp_common.cuh"

namespace pp {

// Ascending key order = descending logit, ties by ascending expert index.
PP_DEVINL unsigned long long rank_key(float g, int j) {
    unsigned u = __float_as_uint(g);
    if ((u << 1) == 0u) u = 0u;  // -0 and +0 are the same logit
    const unsigned ord = (u & 0x80000000u) ? ~u : (u | 0x80000000u);  // ascending in g
    return ((unsigned long long)(~ord) << 32) | (unsigned)j;
}

PP_DEVINL float key_logit(unsigned long long k) {
    const unsigned ord = ~(unsigned)(k >> 32);
    const unsigned u = (ord & 0x80000000u) ? (ord & 0x7fffffffu) : ~ord;
    return __uint_as_float(u);
}

PP_DEVINL int key_index(unsigned long long k) { return (int)(unsigned)(k & 0xffffffffull); }

// One in-lane compare-exchange stage (partner slot s | STRIDE).
template <int S, int STRIDE>
PP_DEVINL void inlane_stage(unsigned long long (&key)[S], int lane, int size) {
    if constexpr (STRIDE < S) {
#pragma unroll
        for (int s = 0; s < S; s++) {
            if ((s & STRIDE) == 0) {
                const int s2 = s | STRIDE;
                const bool asc = ((lane * S + s) & size) == 0;
                const unsigned long long a = key[s], b = key[s2];
                const bool sw = asc ? (a > b) : (a < b);
                key[s] = sw ? b : a;
                key[s2] = sw ? a : b;
            }
        }
    }
}

// Bitonic sort of the warp's 32*S keys into ascending order.  The stage
// loops stay rolled (only the per-lane slot loop is unrolled): the network
// is executed once per token, so compact code that stays in the
// instruction cache beats straight-line code.
template <int S>
PP_DEVINL void warp_bitonic_sort(unsigned long long (&key)[S]) {
    const int lane = threadIdx.x & 31;
#pragma unroll 1
    for (int size = 2; size <= 32 * S; size <<= 1) {
#pragma unroll 1
        for (int stride = size >> 1; stride > 0; stride >>= 1) {
            if (stride >= S) {
                const int ls = stride / S;
                const bool lower = (lane & ls) == 0;
#pragma unroll
                for (int s = 0; s < S; s++) {
                    const bool asc = ((lane * S + s) & size) == 0;
                    const unsigned long long o = __shfl_xor_sync(kFull, key[s], ls);
                    const bool take_min = lower == asc;
                    const unsigned long long lo = key[s] < o ? key[s] : o;
                    const unsigned long long hi = key[s] < o ? o : key[s];
                    key[s] = take_min ? lo : hi;
                }
            } else if (stride == 4) {
                inlane_stage<S, 4>(key, lane, size);
            } else if (stride == 2) {
                inlane_stage<S, 2>(key, lane, size);
            } else {
                inlane_stage<S, 1>(key, lane, size);
            }
        }
    }
}

// The rule parameter as the kernels take it (rule_kernel_param on the host):
// MIN_PREFIX / PAPER the mass budget p; TOPK the count k (an integer in
// [1, E]); LTE the smallest activated fp32 logit (Eq. lte_hard_set:
// sigmoid(g) > delta  <=>  g > ln(delta / (1 - delta))).

// Selection of one token by one warp.  `load(j)` returns logit j (j < E).
// Returns the activated count k (warp-uniform); 0 when a logit is not finite
// (then *finite_out = false).  key[] is left sorted (see file comment).
template <int S, typename Load>
PP_DEVINL int warp_select(Load load, int E, float p, int rule, unsigned long long (&key)[S],
                          bool* finite_out) {
    const int lane = threadIdx.x & 31;
    bool fin = true;
#pragma unroll
    for (int s = 0; s < S; s++) {
        const int j = lane + 32 * s;
        if (j < E) {
            const float v = load(j);
            fin = fin && isfinite(v);
            key[s] = rank_key(v, j);
        } else {
            key[s] = ~0ull;  // padding sorts after every real key
        }
    }
    const bool all_finite = __all_sync(kFull, fin);
    *finite_out = all_finite;
    if (!all_finite) return 0;

    warp_bitonic_sort<S>(key);

    if (rule == PP_SEL_TOPK) return min(E, (int)p);  // the first k ranks
    if (rule == PP_SEL_LTE) {  // the logits at or above the bound form a prefix of the order
        int n = 0;
#pragma unroll
        for (int s = 0; s < S; s++) n += __popc(__ballot_sync(kFull, lane * S + s < E && key_logit(key[s]) >= p));
        return n;
    }

    const float m = key_logit(__shfl_sync(kFull, key[0], 0));  // rank 1 holds max g
    double pre[S];
    double acc = 0.0;
#pragma unroll
    for (int s = 0; s < S; s++) {
        const int r = lane * S + s;
        const float e = (r < E) ? expf(key_logit(key[s]) - m) : 0.0f;
        acc += (double)e;
        pre[s] = acc;
    }
    double incl = acc;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const double v = __shfl_up_sync(kFull, incl, o);
        if (lane >= o) incl += v;
    }
    double excl = __shfl_up_sync(kFull, incl, 1);
    if (lane == 0) excl = 0.0;
    const double Z = __shfl_sync(kFull, incl, 31);
    const double thr = (double)p * Z;
    int below = 0;  // #{ranks i : S_i < p}
#pragma unroll
    for (int s = 0; s < S; s++) {
        const int r = lane * S + s;
        const bool b = (r < E) && (excl + pre[s] < thr);
        below += __popc(__ballot_sync(kFull, b));
    }
    if (p >= 1.0f) return E;  // every expert (warm-up reading)
    if (rule == PP_SEL_PAPER) return below > 1 ? below : 1;
    return below + 1 < E ? below + 1 : E;
}

// Gate weight of the expert at a sorted key (Eq. moe_output).
PP_DEVINL float gate_of(int gate_mode, unsigned long long k) {
    return gate_mode == PP_GATE_NONE ? 1.0f : sigmoidf_(key_logit(k));
}

// ---------------------------------------------------------------------------
// CTA-parallel selection of one token (used where a single token's latency
// matters).  Thread j owns expert j (E <= blockDim.x <= 256).  Instead of
// sorting, every thread sums the exponentials of the experts ranked ahead of
// it: A_j = S_{r_j - 1}, the exclusive prefix mass at its rank r_j in the
// descending order, with equal logits ordered by index: expert i is ahead
// of j when its order key D_i (32 bits, smaller for a larger logit) is below
// D_j, or equal to it with i < j.  Candidates of lower index are compared
// with D_j + 1 and the others with D_j, so the count loop stays in 32-bit
// compares.  The
// exponentials e_j = exp(g_j - max g) (fp32) are summed as exact 2^-31
// fixed-point integers and the cut compares masses with p * Z exactly in
// integers, so the only rounding is that of the fp32 exponentials.
//   MIN_PREFIX: j activated <=> A_j == 0 (rank 0)  or  A_j       <  p Z
//   PAPER:      j activated <=> A_j == 0 (rank 0)  or  A_j + U_j <  p Z
// (the top expert has e = 1, U = 2^31 > 0, so A_j == 0 exactly at rank 0;
// A is non-decreasing along the order, so both sets are prefixes of it).
// TOPK counts with U = 1 for every expert, so A_j is the rank of j:
//   TOPK:       j activated <=> A_j < k
// and LTE needs no count at all:
//   LTE:        j activated <=> g_j >= the bound.

struct CtaSelScratch {
    // order keys D[0..255] and fixed-point exponentials U[256..511] (e * 2^31)
    // for the top-k count; the (D, index) keys of the mass-cut candidates;
    // after the count, the activated (D, index) keys
    __align__(16) uint32_t DU[2 * kMaxExperts];
    float fred[8];
    unsigned long long ured[8];
    int wcnt[8];
    __align__(16) uint32_t cu[kMaxExperts];  // U of each compacted candidate (keys in DU)
    uint8_t flag[kMaxExperts];               // activated experts of the candidate path
    int ncand;
};


PP_DEVINL uint32_t desc_key(float g) {
    unsigned u = __float_as_uint(g);
    if ((u << 1) == 0u) u = 0u;
    const unsigned ord = (u & 0x80000000u) ? ~u : (u | 0x80000000u);
    return ~ord;
}

// Largest integer M with M * 2^sh < p_mant * Z, for p = p_mant * 2^-sh in
// (0, 1); returns -1 (as a flag) when no prefix can be below p Z.
PP_DEVINL long long prefix_threshold(float p, unsigned long long Z) {
    if (!(p > 0.0f)) return -1;
    const unsigned bits = __float_as_uint(p);
    const unsigned ex = (bits >> 23) & 0xffu;
    const unsigned long long mant = ex ? ((bits & 0x7fffffu) | 0x800000u) : (bits & 0x7fffffu);
    const int sh = ex ? 150 - (int)ex : 149;
    const unsigned long long rhs = mant * Z;  // < 2^24 * 2^39
    if (rhs == 0ull) return -1;
    if (sh >= 64) return 0;  // only an empty prefix (mass 0) is below p Z
    return (long long)((rhs - 1ull) >> sh);
}

// Returns the activated count k (CTA-uniform).  On return: *sel = whether
// expert j (= threadIdx.x) is activated, *gval = its logit and, when
// want_rank, *rank = its rank for activated experts (the activated experts
// hold ranks 0 .. k-1); *rank is -1 otherwise.  All threads of the CTA (8
// warps) must call it with the same want_rank.
template <typename Load>
PP_DEVINL int cta_select_fn(Load load, int E, float p, int rule, bool want_rank, CtaSelScratch& sc,
                            unsigned* status, bool* sel, int* rank, float* gval) {
    const int j = threadIdx.x;
    const int lane = j & 31, warp = j >> 5;
    const bool valid = j < E;
    const float g = valid ? load(j) : -INFINITY;
    *gval = g;
    *rank = -1;
    sc.flag[j] = 0;  // read back after the count (a later barrier orders it)
    const bool fin = !valid || isfinite(g);
    if (!__syncthreads_and(fin)) {
        if (j == 0) record_status(status, PP_ERR_NONFINITE);
        *sel = false;
        return 0;
    }
    // max logit: warp shuffles, then the 8 warp maxima read as two vectors
    float m = g;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) m = fmaxf(m, __shfl_xor_sync(kFull, m, o));
    if (lane == 0) sc.fred[warp] = m;
    __syncthreads();
    {
        const float4 a = *reinterpret_cast<const float4*>(&sc.fred[0]);
        const float4 b = *reinterpret_cast<const float4*>(&sc.fred[4]);
        m = fmaxf(fmaxf(fmaxf(a.x, a.y), fmaxf(a.z, a.w)), fmaxf(fmaxf(b.x, b.y), fmaxf(b.z, b.w)));
    }
    // fixed-point exponentials and their sum Z
    const float e = valid ? expf(g - m) : 0.0f;
    const uint32_t U = valid ? (rule == PP_SEL_TOPK ? 1u : __float2uint_rn(e * 2147483648.0f)) : 0u;
    const uint32_t D = valid ? desc_key(g) : 0xffffffffu;  // a finite logit never gives all ones
    uint32_t* sD = sc.DU;
    uint32_t* sU = sc.DU + kMaxExperts;
    unsigned long long* sK = reinterpret_cast<unsigned long long*>(sc.DU);
    if (rule == PP_SEL_TOPK) {
        sD[j] = D;
        sU[j] = U;
    } else {
        // padding of the candidate list (a key that is never ahead)
        sK[j] = ~0ull;
        sc.cu[j] = 0u;
        if (j == 0) sc.ncand = 0;
    }
    unsigned long long z = U;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) z += __shfl_xor_sync(kFull, z, o);
    if (lane == 0) sc.ured[warp] = z;
    __syncthreads();
    unsigned long long Z;
    {
        const ulonglong2* v = reinterpret_cast<const ulonglong2*>(sc.ured);
        const ulonglong2 a = v[0], b = v[1], c = v[2], d2 = v[3];
        Z = (a.x + a.y) + (b.x + b.y) + (c.x + c.y) + (d2.x + d2.y);
    }
    bool on = false, counted = false, filtered = false;
    if (rule == PP_SEL_LTE) {
        on = counted = valid && g >= p;
    } else if (rule != PP_SEL_TOPK && p >= 1.0f) {
        on = counted = valid;  // every expert (warm-up reading)
    } else if (rule == PP_SEL_TOPK) {
        // exclusive rank by counting, four independent accumulator chains;
        // candidates [0, w0) have a lower index than every thread of this
        // warp, [w0, w1) are the warp's own experts, [w1, E) have a higher
        // index
        unsigned long long m0 = 0, m1 = 0, m2 = 0, m3 = 0;
        const int w0 = warp * 32, w1 = min(E, w0 + 32);
        if (w0 < E) {  // warps without an expert skip the count
            const uint32_t thrB = D + 1u, thrA = D;
            // candidates [i0, i1) against threshold th (or, in the warp's own
            // range, th for index >= j and th + 1 below j); 16 candidates are
            // loaded before any of them is compared, so the shared-memory
            // latency is paid once per 16
            auto accum = [&](int i0, int i1, uint32_t th, bool own) {
                int i = i0;
                for (; i + 16 <= i1; i += 16) {
                    uint4 d4[4], u4[4];
#pragma unroll
                    for (int k = 0; k < 4; k++) {
                        d4[k] = *reinterpret_cast<const uint4*>(&sD[i + 4 * k]);
                        u4[k] = *reinterpret_cast<const uint4*>(&sU[i + 4 * k]);
                    }
#pragma unroll
                    for (int k = 0; k < 4; k++) {
                        const int b = i + 4 * k;
                        const uint32_t t0 = own && b + 0 < j ? th + 1u : th, t1 = own && b + 1 < j ? th + 1u : th;
                        const uint32_t t2 = own && b + 2 < j ? th + 1u : th, t3 = own && b + 3 < j ? th + 1u : th;
                        m0 += d4[k].x < t0 ? (unsigned long long)u4[k].x : 0ull;
                        m1 += d4[k].y < t1 ? (unsigned long long)u4[k].y : 0ull;
                        m2 += d4[k].z < t2 ? (unsigned long long)u4[k].z : 0ull;
                        m3 += d4[k].w < t3 ? (unsigned long long)u4[k].w : 0ull;
                    }
                }
                for (; i < i1; i++) m0 += sD[i] < (own && i < j ? th + 1u : th) ? (unsigned long long)sU[i] : 0ull;
            };
            accum(0, w0, thrB, false);
            accum(w0, w1, thrA, true);
            accum(w1, E, thrA, false);
        }
        const unsigned long long ahead = (m0 + m1) + (m2 + m3);
        on = counted = valid && ahead < (unsigned long long)(int)p;
    } else {
        // Cumulative-mass cut.  Only experts near the top of the order can
        // be activated: the mass at or behind an activated j exceeds
        // (1 - p) Z and consists of at most E exponentials no larger than
        // e_j (up to the 2-ulp error of expf), so e_j > (1 - p) Z / E.  The
        // candidates are the experts with g_j - m >= ln of half that bound
        // (a slack of ln 2 for the roundings); the test is monotone in g, so
        // they form a prefix of the order, every expert ahead of a
        // candidate is one, and a candidate's exclusive prefix mass A_j is
        // summed over the candidates alone.  Below a bound of 20 * 2^-31
        // every expert is a candidate.
        filtered = true;
        // the bound needs no rounding care (slack ln 2): fast log and divide
        const float Bm = __fdividef((1.0f - fmaxf(p, 0.0f)) * ((float)Z * (1.0f / 2147483648.0f)), (float)E);
        const float Lc = Bm >= 20.0f / 2147483648.0f ? __logf(0.5f * Bm) : -INFINITY;
        const bool cand = valid && (g - m) >= Lc;
        const long long thr = prefix_threshold(p, Z);
        // compaction in arrival order through a warp-aggregated shared
        // counter; the key (D, index) carries the tie-break, and the slots
        // past the last candidate keep the padding written before the
        // previous barrier
        const unsigned bal = __ballot_sync(kFull, cand);
        int wbase = 0;
        if (lane == 0 && bal) wbase = atomicAdd(&sc.ncand, __popc(bal));
        wbase = __shfl_sync(kFull, wbase, 0);
        if (cand) {
            const int q = wbase + __popc(bal & ((1u << lane) - 1u));
            sK[q] = ((unsigned long long)D << 32) | (unsigned)j;
            sc.cu[q] = U;
        }
        __syncthreads();
        const int nc = sc.ncand;
        // nt = 2^lg threads per candidate (aligned lane groups), each summing
        // a contiguous run of the candidates, four at a time
        const int lg = nc <= 16 ? 4 : nc <= 32 ? 3 : nc <= 64 ? 2 : nc <= 128 ? 1 : 0;
        const int nt = 1 << lg;
        const int q = j >> lg, part = j & (nt - 1);
        unsigned long long a0 = 0ull, a1 = 0ull;
        if (q < nc) {
            const unsigned long long Kq = sK[q];
            const int nv = (nc + 3) >> 2, per = (nv + nt - 1) >> lg;
            const int v1 = min(nv, (part + 1) * per);
            const ulonglong2* k2 = reinterpret_cast<const ulonglong2*>(sK);
            const uint4* u4p = reinterpret_cast<const uint4*>(sc.cu);
            for (int v = part * per; v < v1; v++) {
                const ulonglong2 ka = k2[2 * v], kb = k2[2 * v + 1];
                const uint4 u4 = u4p[v];
                a0 += ka.x < Kq ? (unsigned long long)u4.x : 0ull;
                a1 += ka.y < Kq ? (unsigned long long)u4.y : 0ull;
                a0 += kb.x < Kq ? (unsigned long long)u4.z : 0ull;
                a1 += kb.y < Kq ? (unsigned long long)u4.w : 0ull;
            }
        }
        unsigned long long a = a0 + a1;
        for (int o = 1; o < nt; o <<= 1) a += __shfl_xor_sync(kFull, a, o);
        if (q < nc && part == 0) {
            const unsigned long long mass = rule == PP_SEL_PAPER ? a + sc.cu[q] : a;
            counted = a == 0ull || (thr >= 0 && mass <= (unsigned long long)thr);
            if (counted) sc.flag[(unsigned)sK[q] & 0xffu] = 1;
        }
    }
    const int k = __syncthreads_count(counted);  // also: every thread is done reading sD, sU
    if (filtered) on = valid && sc.flag[j] != 0;
    *sel = on;
    if (want_rank) {
        // rank of an activated expert = activated keys (D, index) below its
        // own; the activated keys are compacted into the scratch first
        const unsigned long long key = ((unsigned long long)D << 32) | (unsigned)j;
        const unsigned bal = __ballot_sync(kFull, on);
        if (lane == 0) sc.wcnt[warp] = __popc(bal);
        __syncthreads();
        int base = 0;
        for (int w = 0; w < warp; w++) base += sc.wcnt[w];
        if (on) sK[base + __popc(bal & ((1u << lane) - 1u))] = key;
        __syncthreads();
        if (on) {
            int r = 0;
            for (int i = 0; i < k; i++) r += sK[i] < key ? 1 : 0;
            *rank = r;
        }
        __syncthreads();  // the scratch is reused by the next call
    }
    return k;
}

// ---------------------------------------------------------------------------
// Cumulative-mass cut of one token (MIN_PREFIX or PAPER with p < 1) by the
// whole CTA in three barriers, for the fused decode kernel, where every
// instruction of this serial step is latency.  Thread j holds logit j.  Same
// arithmetic as cta_select_fn: fp32 max-shifted exponentials summed as exact
// 2^-31 fixed-point integers; the candidates (a prefix of the order) each get
// their exclusive prefix mass A and rank counted over the candidates ahead of
// them; then
//   MIN_PREFIX: activated <=> A == 0 or A      <= M
//   PAPER:      activated <=> A == 0 or A + U  <= M
// with M = prefix_threshold(p, Z) (the largest integer below p Z).  An
// activated expert carries more than (1 - p) Z / E of the mass (the mass at
// or behind it exceeds (1 - p) Z and holds at most E exponentials no larger
// than its own), so the candidates are the experts with
// g - max >= ln((1 - p) Z' / (2 E)), where Z' is Z to within a few parts in
// 10^7 (each warp's sum of exp(g - its own max) in 2^-24 fixed point,
// rescaled to the global max): any Z' below 2 Z keeps every activated
// expert, and the slack of ln 2 also covers the fast log.
//   barrier 1: warp maxima (order keys) and approximate sums, non-finite flag
//   barrier 2: exact warp sums of the fixed-point exponentials; candidates
//              compacted by one shared atomic per warp
//   barrier 3: the activated count
struct WarpCand {
    unsigned long long key;  // (descending-logit key << 32) | expert index
    uint32_t U;              // fixed-point exponential
    float g;                 // logit
};

struct CutShared {
    uint32_t wmin[8];  // per warp: smallest order key (its max logit)
    uint32_t zw[8];    // per warp: sum of exp(g - its max) in 2^-24 units
    uint32_t zhi[8];   // per warp: sums of the exponentials' high and low 16 bits
    uint32_t zlo[8];
    int nc;            // candidates
};

PP_DEVINL float desc_key_logit(uint32_t D) {
    const unsigned ord = ~D;
    return __uint_as_float((ord & 0x80000000u) ? (ord & 0x7fffffffu) : ~ord);
}

// Barriers of a group of nt threads (whole warps) with barrier id `id`
// (id 0 with the whole CTA is __syncthreads).
PP_DEVINL void group_bar(int id, int nt) { asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(nt) : "memory"); }
PP_DEVINL bool group_bar_or(int id, int nt, bool v) {
    unsigned r;
    asm volatile(
        "{\n\t.reg .pred pi, po;\n\t"
        "setp.ne.u32 pi, %1, 0;\n\t"
        "bar.red.or.pred po, %2, %3, pi;\n\t"
        "selp.u32 %0, 1, 0, po;\n\t}"
        : "=r"(r)
        : "r"((unsigned)v), "r"(id), "r"(nt)
        : "memory");
    return r != 0u;
}
PP_DEVINL int group_bar_count(int id, int nt, bool v) {
    unsigned r;
    asm volatile(
        "{\n\t.reg .pred pi;\n\t"
        "setp.ne.u32 pi, %1, 0;\n\t"
        "bar.red.popc.u32 %0, %2, %3, pi;\n\t}"
        : "=r"(r)
        : "r"((unsigned)v), "r"(id), "r"(nt)
        : "memory");
    return (int)r;
}

// Every thread of a group of nt = 32 w threads (w <= 8 whole warps, nt >= E)
// calls, with the group's barrier id; thread j < E of the group passes logit
// j.  cand: nt entries of scratch (shared memory); sc: the group's own.  For
// every activated expert one thread calls on(rank, expert, logit); every
// thread calls mid() after barrier 2.  Returns the activated count k, or 0
// with PP_ERR_NONFINITE recorded when a logit is not finite.
template <typename On, typename Mid>
PP_DEVINL int group_mass_cut(float g, int E, float p, int rule, CutShared& sc, WarpCand* cand, unsigned* status,
                             int bid, int nt, On on, Mid mid) {
    const int j = threadIdx.x & (nt - 1), lane = j & 31, warp = j >> 5, nw = nt >> 5;
    const bool valid = j < E;
    const bool fin = !valid || isfinite(g);
    const uint32_t D = valid && fin ? desc_key(g) : 0xffffffffu;
    const uint32_t wmin = __reduce_min_sync(kFull, D);
    const float mw = desc_key_logit(wmin);
    const uint32_t zw = __reduce_add_sync(kFull, valid && fin ? __float2uint_rn(expf(g - mw) * 16777216.0f) : 0u);
    if (lane == 0) {
        sc.wmin[warp] = wmin;
        sc.zw[warp] = zw;
    }
    if (j == 0) sc.nc = 0;
    if (group_bar_or(bid, nt, !fin)) {
        if (j == 0) record_status(status, PP_ERR_NONFINITE);
        return 0;
    }
    uint32_t dmin = 0xffffffffu;  // (loops unrolled to 8 so that the loads issue together)
#pragma unroll
    for (int w = 0; w < 8; w++)
        if (w < nw) dmin = min(dmin, sc.wmin[w]);
    const float m = desc_key_logit(dmin);
    // sum of exp(g - m) to a few parts in 10^7: lane w < nw rescales warp w's
    // sum, three shuffles add the (up to eight) terms
    float zapprox = 0.0f;
    if (lane < nw) {
        const uint32_t dw = sc.wmin[lane];
        if (dw != 0xffffffffu) zapprox = (float)sc.zw[lane] * (1.0f / 16777216.0f) * expf(desc_key_logit(dw) - m);
    }
    zapprox += __shfl_xor_sync(kFull, zapprox, 4);
    zapprox += __shfl_xor_sync(kFull, zapprox, 2);
    zapprox += __shfl_xor_sync(kFull, zapprox, 1);
    zapprox = __shfl_sync(kFull, zapprox, 0);
    const uint32_t U = valid ? __float2uint_rn(expf(g - m) * 2147483648.0f) : 0u;
    const float Bm = __fdividef((1.0f - fmaxf(p, 0.0f)) * zapprox, (float)E);
    const float Lc = Bm >= 20.0f / 2147483648.0f ? __logf(0.5f * Bm) : -INFINITY;
    const bool c = valid && (g - m) >= Lc;
    const unsigned bal = __ballot_sync(kFull, c);
    int base = 0;
    if (lane == 0 && bal) base = atomicAdd(&sc.nc, __popc(bal));
    base = __shfl_sync(kFull, base, 0);
    if (c) cand[base + __popc(bal & ((1u << lane) - 1u))] = WarpCand{((unsigned long long)D << 32) | (unsigned)j, U, g};
    const uint32_t hi = __reduce_add_sync(kFull, U >> 16), lo = __reduce_add_sync(kFull, U & 0xffffu);
    if (lane == 0) {
        sc.zhi[warp] = hi;
        sc.zlo[warp] = lo;
    }
    group_bar(bid, nt);
    mid();
    unsigned long long Z = 0ull;
#pragma unroll
    for (int w = 0; w < 8; w++)
        if (w < nw) Z += ((unsigned long long)sc.zhi[w] << 16) + sc.zlo[w];
    const int nc = sc.nc;
    const long long thr = prefix_threshold(p, Z);
    // gs threads per candidate (aligned lane groups), each summing a
    // contiguous run of the list.  nc <= E <= nt and gs * nc <= nt, so a
    // thread takes one candidate at most.
    int lg = 0;
    while (lg < 5 && (nc << (lg + 1)) <= nt) lg++;
    const int gs = 1 << lg;
    const int q = j >> lg, part = j & (gs - 1);
    const bool mine = q < nc;
    const WarpCand cq = cand[mine ? q : 0];
    const int per = (nc + gs - 1) >> lg;
    const int i0 = min(nc, part * per), i1 = min(nc, i0 + per);
    unsigned long long A0 = 0ull, A1 = 0ull;
    int r0 = 0, r1 = 0;
    int i = i0;
    for (; i + 2 <= i1; i += 2) {
        const WarpCand c0 = cand[i], c1 = cand[i + 1];
        const bool a0 = c0.key < cq.key, a1 = c1.key < cq.key;
        A0 += a0 ? (unsigned long long)c0.U : 0ull;
        A1 += a1 ? (unsigned long long)c1.U : 0ull;
        r0 += a0;
        r1 += a1;
    }
    if (i < i1) {
        const WarpCand c0 = cand[i];
        const bool a0 = c0.key < cq.key;
        A0 += a0 ? (unsigned long long)c0.U : 0ull;
        r0 += a0;
    }
    unsigned long long A = A0 + A1;
    int r = r0 + r1;
    for (int o = 1; o < gs; o <<= 1) {
        A += __shfl_xor_sync(kFull, A, o);
        r += __shfl_xor_sync(kFull, r, o);
    }
    const unsigned long long mass = rule == PP_SEL_PAPER ? A + cq.U : A;
    const bool act = mine && part == 0 && (A == 0ull || (thr >= 0 && mass <= (unsigned long long)thr));
    if (act) on(r, (int)(unsigned)(cq.key & 0xffffffffull), cq.g);
    return group_bar_count(bid, nt, act);
}

// The whole CTA (8 warps) on one token.
template <typename On, typename Mid>
PP_DEVINL int cta_mass_cut(float g, int E, float p, int rule, CutShared& sc, WarpCand* cand, unsigned* status, On on,
                           Mid mid) {
    return group_mass_cut(g, E, p, rule, sc, cand, status, 0, 256, on, mid);
}

// The rank-order selection row of one token from cta_select_fn's results
// (called by every thread j < E): activated experts at their ranks, -1 and
// gate 0 in the slots k .. E-1.
PP_DEVINL void write_selection_row(int32_t* ids, float* gates, int j, int E, int k, bool on, int r, float gv) {
    if (on) {
        ids[r] = j;
        gates[r] = gv;
    }
    if (j >= k && j < E) {
        ids[j] = -1;
        gates[j] = 0.0f;
    }
}

}  // namespace pp
