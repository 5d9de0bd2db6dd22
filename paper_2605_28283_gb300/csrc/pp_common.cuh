// Device helpers shared by the PrunePath kernels (sm_103a).
//
// Inline PTX wrappers for mbarriers, bulk and tensor TMA copies, proxy
// fences and the global timer; a bounded mbarrier wait; tagged 64-bit words
// for handing values between the CTAs of one co-resident (cooperative) grid
// without a grid barrier; bf16 helpers.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "prunepath.h"

#define PP_DEVINL __device__ __forceinline__

namespace pp {

constexpr int kDExpert = 64;      // d_e, the expert width this library is built for
constexpr int kMaxExperts = 256;  // E limit (the warp sort holds 8 keys per lane)
constexpr int kMaxD = 8192;
constexpr unsigned kFull = 0xffffffffu;

// ------------------------------------------------------------------ control
// The first 1280 bytes of every workspace.
constexpr int kMaxGrid = 256;  // CTAs of a fused decode launch (one per SM)
struct Control {
    unsigned status;           // sticky pp_status of the device side
    unsigned wait_flag;        // never written: target of pp_debug_wait_timeout
    unsigned pad[62];
    unsigned epoch[kMaxGrid];  // launches of the fused decode kernel seen by CTA b
};
static_assert(sizeof(Control) == 1280, "control block is 1280 bytes");

PP_DEVINL void record_status(unsigned* status, pp_status s) {
    // first error wins; later ones do not overwrite it
    atomicCAS(status, 0u, (unsigned)s);
}

PP_DEVINL uint64_t globaltimer_ns() {
    uint64_t t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}

// ----------------------------------------------------------------- mbarrier
PP_DEVINL uint32_t smem_u32(const void* p) { return (uint32_t)__cvta_generic_to_shared(p); }

PP_DEVINL void mbar_init(uint64_t* bar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count));
}

PP_DEVINL void fence_mbar_init() { asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory"); }

PP_DEVINL void mbar_arrive_expect_tx(uint64_t* bar, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)),
                 "r"(bytes)
                 : "memory");
}

PP_DEVINL void mbar_arrive(uint64_t* bar) {
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}

PP_DEVINL bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(smem_u32(bar)), "r"(parity)
        : "memory");
    return ok != 0;
}

// Wait for the phase with the given parity to complete, for at most
// limit_ns.  On expiry records PP_ERR_TIMEOUT and returns false.  A wait
// that has lasted over 1 ms also gives up as soon as another wait has
// recorded an error, so one failure cannot chain into many full timeouts.
// The bounded loop is a separate (not inlined) function: kernels that run
// once per launch are bound by instruction fetch, so every call site keeps
// only the first try_wait inline.
static __device__ __noinline__ bool mbar_wait_slow(uint64_t* bar, uint32_t parity, unsigned* status,
                                                   uint64_t limit_ns) {
    const uint64_t t0 = globaltimer_ns();
    while (true) {
        if (mbar_try_wait(bar, parity)) return true;
        const uint64_t dt = globaltimer_ns() - t0;
        if (dt > limit_ns) {
            record_status(status, PP_ERR_TIMEOUT);
            return false;
        }
        if (dt > 1000000ull && *reinterpret_cast<volatile unsigned*>(status) != 0u) return false;
    }
}

PP_DEVINL bool mbar_wait(uint64_t* bar, uint32_t parity, unsigned* status, uint64_t limit_ns) {
    if (mbar_try_wait(bar, parity)) return true;
    return mbar_wait_slow(bar, parity, status, limit_ns);
}

// -------------------------------------------------------------------- TMA
// 1-D bulk copy global -> shared, completion counted in bytes on `bar`.
// src, dst 16-byte aligned, bytes a multiple of 16.
PP_DEVINL void bulk_g2s(void* dst, const void* src, uint32_t bytes, uint64_t* bar) {
    asm volatile(
        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
            smem_u32(dst)),
        "l"(src), "r"(bytes), "r"(smem_u32(bar))
        : "memory");
}

// 2-D tiled tensor copy global -> shared.  c0 is the inner (contiguous)
// coordinate; c0 * element size must be a multiple of 16 bytes.
PP_DEVINL void tma_load_2d(void* dst, const CUtensorMap* map, int c0, int c1, uint64_t* bar) {
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes [%0], [%1, "
        "{%2, %3}], [%4];" ::"r"(smem_u32(dst)),
        "l"(reinterpret_cast<uint64_t>(map)), "r"(c0), "r"(c1), "r"(smem_u32(bar))
        : "memory");
}

// 2-D tiled prefetch of a tensor-map box into L2 (no shared memory).
PP_DEVINL void tma_prefetch_2d(const CUtensorMap* map, int c0, int c1) {
    asm volatile("cp.async.bulk.prefetch.tensor.2d.L2.global.tile [%0, {%1, %2}];" ::"l"(reinterpret_cast<uint64_t>(map)),
                 "r"(c0), "r"(c1)
                 : "memory");
}

// Programmatic dependent launch: wait until the preceding grid on the stream
// has completed and its memory is visible (no-op when launched without the
// attribute); allow the next grid on the stream to start launching.
PP_DEVINL void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
PP_DEVINL void pdl_launch_dependents() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }

// Order this thread's earlier generic-proxy shared-memory accesses before
// later async-proxy (TMA) accesses of the same memory.
PP_DEVINL void fence_proxy_async_smem() { asm volatile("fence.proxy.async.shared::cta;" ::: "memory"); }

PP_DEVINL void named_bar_sync(int id, int nthreads) {
    asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(nthreads) : "memory");
}

// ---------------------------------------------------------- tagged words
PP_DEVINL unsigned ld_acquire_gpu(const unsigned* p) {
    unsigned v;
    asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    return v;
}

// A value handed from one CTA to others of the same launch travels with the
// launch's tag in one 64-bit word, (tag << 32) | bits(value).  A 64-bit store
// is single-copy atomic, so a reader that sees the tag sees the value: no
// flag, fence or grid barrier is needed, and each reader waits only for the
// words it uses.  Tags change from launch to launch (a launch never takes its
// predecessor's words for current) and are not 0, the value of a zeroed
// workspace, before 2^32 - 1 launches.
PP_DEVINL void st_tagged(unsigned long long* p, unsigned tag, float v) {
    const unsigned long long w = ((unsigned long long)tag << 32) | __float_as_uint(v);
    asm volatile("st.relaxed.gpu.global.u64 [%0], %1;" ::"l"(p), "l"(w) : "memory");
}

PP_DEVINL unsigned long long ld_relaxed_u64(const unsigned long long* p) {
    unsigned long long v;
    asm volatile("ld.relaxed.gpu.global.u64 %0, [%1];" : "=l"(v) : "l"(p) : "memory");
    return v;
}

PP_DEVINL void ld_relaxed_v2(const unsigned long long* p, unsigned long long& a, unsigned long long& b) {
    asm volatile("ld.relaxed.gpu.global.v2.u64 {%0, %1}, [%2];" : "=l"(a), "=l"(b) : "l"(p) : "memory");
}

PP_DEVINL unsigned word_tag(unsigned long long w) { return (unsigned)(w >> 32); }
PP_DEVINL float word_value(unsigned long long w) { return __uint_as_float((unsigned)w); }

// Pause between two polls of the same words: without it, every SM re-reading
// a handful of L2 lines back to back slows the stores and loads of the CTAs
// that are still working.
constexpr unsigned kPollBackoffNs = 64;

// Bookkeeping of a bounded poll: true when the caller should stop polling,
// after limit_ns (recording PP_ERR_TIMEOUT) or, past 1 ms, as soon as another
// wait has recorded an error.
PP_DEVINL bool poll_give_up(uint64_t& t0, unsigned* status, uint64_t limit_ns) {
    const uint64_t now = globaltimer_ns();
    if (t0 == 0) {
        t0 = now;
        return false;
    }
    const uint64_t dt = now - t0;
    if (dt > limit_ns) {
        record_status(status, PP_ERR_TIMEOUT);
        return true;
    }
    return dt > 1000000ull && *reinterpret_cast<volatile unsigned*>(status) != 0u;
}

// Value of the tagged word at p once it carries `tag` (bounded; on giving up
// the stale value is returned and the status says why).
PP_DEVINL float wait_tagged(const unsigned long long* p, unsigned tag, unsigned* status, uint64_t limit_ns) {
    unsigned long long w = ld_relaxed_u64(p);
    uint64_t t0 = 0;
    while (word_tag(w) != tag && !poll_give_up(t0, status, limit_ns)) {
        __nanosleep(kPollBackoffNs);
        w = ld_relaxed_u64(p);
    }
    return word_value(w);
}

// ------------------------------------------------------------------- bf16
PP_DEVINL float bf16lo(uint32_t w) { return __uint_as_float(w << 16); }
PP_DEVINL float bf16hi(uint32_t w) { return __uint_as_float(w & 0xffff0000u); }

// Element access for the two storage types.
template <typename TW>
struct Elem;

template <>
struct Elem<float> {
    static constexpr int kPer16B = 4;
    PP_DEVINL static void unpack(const uint4& v, float* f) {
        f[0] = __uint_as_float(v.x);
        f[1] = __uint_as_float(v.y);
        f[2] = __uint_as_float(v.z);
        f[3] = __uint_as_float(v.w);
    }
    PP_DEVINL static void store(void* base, size_t i, float v) { reinterpret_cast<float*>(base)[i] = v; }
    PP_DEVINL static uint4 pack(const float* f) {
        return make_uint4(__float_as_uint(f[0]), __float_as_uint(f[1]), __float_as_uint(f[2]), __float_as_uint(f[3]));
    }
};

template <>
struct Elem<__nv_bfloat16> {
    static constexpr int kPer16B = 8;
    PP_DEVINL static void unpack(const uint4& v, float* f) {
        f[0] = bf16lo(v.x);
        f[1] = bf16hi(v.x);
        f[2] = bf16lo(v.y);
        f[3] = bf16hi(v.y);
        f[4] = bf16lo(v.z);
        f[5] = bf16hi(v.z);
        f[6] = bf16lo(v.w);
        f[7] = bf16hi(v.w);
    }
    PP_DEVINL static void store(void* base, size_t i, float v) {
        reinterpret_cast<__nv_bfloat16*>(base)[i] = __float2bfloat16_rn(v);
    }
    // round-to-nearest-even bf16 pairs, low half first
    PP_DEVINL static uint32_t pair(float lo, float hi) {
        const __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
        return *reinterpret_cast<const uint32_t*>(&v);
    }
    PP_DEVINL static uint4 pack(const float* f) {
        return make_uint4(pair(f[0], f[1]), pair(f[2], f[3]), pair(f[4], f[5]), pair(f[6], f[7]));
    }
};

// ------------------------------------------------------------ activations
PP_DEVINL float sigmoidf_(float v) { return 1.0f / (1.0f + expf(-v)); }

// h for one neuron: a = x.W_up row, b = x.W_gate row (Eq. ffn; SiLU gate for
// PP_ACT_SWIGLU, h = relu(a) or the tanh form of GELU otherwise).
PP_DEVINL float act_h(int act, float a, float b) {
    if (act == PP_ACT_SWIGLU) return b / (1.0f + expf(-b)) * a;
    if (act == PP_ACT_RELU) return fmaxf(a, 0.0f);
    const float k0 = 0.7978845608028654f;  // sqrt(2/pi)
    return 0.5f * a * (1.0f + tanhf(k0 * (a + 0.044715f * a * a * a)));
}

PP_DEVINL float warp_sum(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(kFull, v, o);
    return v;
}

PP_DEVINL float warp_max(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(kFull, v, o));
    return v;
}

}  // namespace pp
