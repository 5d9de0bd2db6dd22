// Warp-level cumulative-mass expert selection for one token (PrunePath
// Sec. 3.1: Eq. softmax_prob, the descending order pi, Eq.
// tau_thresh_activate).
//
// One warp holds the token's E <= 32*S logits as 64-bit rank keys, S per
// lane, sorts them with a register bitonic network (in-lane exchanges for
// strides < S, shuffles otherwise), then forms the max-shifted fp32
// exponentials in rank order and their inclusive prefix sums in fp64.  The
// cut compares each prefix with p * Z in fp64.  After the sort lane l holds
// ranks l*S .. l*S+S-1 in key[0..S-1].
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

template <int S>
PP_DEVINL void warp_bitonic_sort(unsigned long long (&key)[S]) {
    const int lane = threadIdx.x & 31;
#pragma unroll
    for (int size = 2; size <= 32 * S; size <<= 1) {
#pragma unroll
        for (int stride = size >> 1; stride > 0; stride >>= 1) {
            if (stride >= S) {
                const int ls = stride / S;
#pragma unroll
                for (int s = 0; s < S; s++) {
                    const int i = lane * S + s;
                    const unsigned long long o = __shfl_xor_sync(kFull, key[s], ls);
                    const bool take_min = ((i & stride) == 0) == ((i & size) == 0);
                    const unsigned long long lo = key[s] < o ? key[s] : o;
                    const unsigned long long hi = key[s] < o ? o : key[s];
                    key[s] = take_min ? lo : hi;
                }
            } else {
#pragma unroll
                for (int s = 0; s < S; s++) {
                    if ((s & stride) == 0) {
                        const int s2 = s | stride;
                        const int i = lane * S + s;
                        const bool asc = (i & size) == 0;
                        const unsigned long long a = key[s], b = key[s2];
                        const bool sw = asc ? (a > b) : (a < b);
                        key[s] = sw ? b : a;
                        key[s2] = sw ? a : b;
                    }
                }
            }
        }
    }
}

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

}  // namespace pp
