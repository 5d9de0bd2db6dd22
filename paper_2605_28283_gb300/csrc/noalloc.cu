// pp_layer_noalloc: the fused decode layer for callers that cannot hand the
// library a workspace.
//
// Some callers cannot call cudaMalloc (or any allocator) at the point where
// they run a layer: a serving runtime that has given all device memory to
// its own pool, a real-time loop that must not take the implicit device
// synchronisation an allocation can cause, or a plug-in host that exposes no
// allocation API to the code it loads.  This entry point runs the same fused
// decode kernel as pp_layer, but its scratch memory (status word, per-CTA
// launch counts, and the tagged router logits and
// gate/up activations the CTAs hand to each other) lives in one file-scope
// device array that every GPU loading the library reserves until the
// process exits.  Nothing is allocated or freed per call.
#include <cstring>
#include <mutex>

#include "pp_common.cuh"
#include "pp_kernels.h"

namespace {

// Limits of the no-allocation variant: up to 4 tokens per call, E <= 256.
constexpr int kNoAllocMaxTokens = 4;
constexpr size_t kCtlBytes = sizeof(pp::Control);  // status word, per-CTA launch counts
constexpr size_t kLogitBytes = (size_t)kNoAllocMaxTokens * pp::kMaxExperts * 8;
constexpr size_t kHBytes = (size_t)pp::kMaxExperts * kNoAllocMaxTokens * pp::kDExpert * 8;
constexpr size_t kScratchBytes = kCtlBytes + kLogitBytes + kHBytes;  // 533,760 bytes
static_assert(kScratchBytes == 533760, "scratch size as documented in prunepath.h");
constexpr uint64_t kTimeoutNs = 2000000000ull;

}  // namespace

// The shared scratch.  Host code only ever uses the address returned by
// cudaGetSymbolAddress for the current device; the symbol itself is a host-side
// stand-in and must never be passed to a kernel.
static __device__ __align__(256) unsigned char g_pp_noalloc_scratch[kScratchBytes];

namespace {

struct DevState {
    bool ready = false;
    unsigned char* scratch = nullptr;  // device address of g_pp_noalloc_scratch
    int sms = 0, cc_major = 0, cc_minor = 0;
    size_t smem_optin = 0;
};

std::mutex g_mu;
DevState g_dev[64];

// Once per device, with that device current: resolve the scratch address and
// cache the device properties.
pp_status device_setup(DevState** out) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return PP_ERR_CUDA;
    std::lock_guard<std::mutex> lock(g_mu);
    DevState& s = g_dev[dev];
    if (!s.ready) {
        void* p = nullptr;
        if (cudaGetSymbolAddress(&p, g_pp_noalloc_scratch) != cudaSuccess || p == nullptr) return PP_ERR_CUDA;
        int v = 0;
        if (cudaDeviceGetAttribute(&s.sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess ||
            cudaDeviceGetAttribute(&s.cc_major, cudaDevAttrComputeCapabilityMajor, dev) != cudaSuccess ||
            cudaDeviceGetAttribute(&s.cc_minor, cudaDevAttrComputeCapabilityMinor, dev) != cudaSuccess ||
            cudaDeviceGetAttribute(&v, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev) != cudaSuccess)
            return PP_ERR_CUDA;
        s.smem_optin = (size_t)v;
        s.scratch = static_cast<unsigned char*>(p);
        s.ready = true;
    }
    *out = &s;
    return PP_OK;
}

bool aligned16(const void* p) { return ((uintptr_t)p & 15u) == 0; }

pp_status check_args(const pp_desc* d, int T, const void* x, const void* Wr, const void* Wg, const void* Wu,
                     const void* Wd, float p, const pp_selection* sel, const void* y) {
    if (!d) return PP_ERR_INVALID_ARG;
    if (d->dtype != PP_F32 && d->dtype != PP_BF16) return PP_ERR_DTYPE;
    if (d->act < PP_ACT_RELU || d->act > PP_ACT_SWIGLU) return PP_ERR_INVALID_ARG;
    if (d->gate != PP_GATE_SIGMOID && d->gate != PP_GATE_NONE) return PP_ERR_INVALID_ARG;
    if (!pp::rule_known(d->rule)) return PP_ERR_INVALID_ARG;
    if (d->d_expert != pp::kDExpert || d->n_experts < 1 || d->n_experts > pp::kMaxExperts) return PP_ERR_SHAPE;
    if ((long long)d->d_ff != (long long)d->n_experts * pp::kDExpert) return PP_ERR_SHAPE;
    const int vec = d->dtype == PP_BF16 ? 8 : 4;
    if (d->d_model < 64 || d->d_model > pp::kMaxD || d->d_model % vec != 0) return PP_ERR_SHAPE;
    if (T < 0 || T > kNoAllocMaxTokens) return PP_ERR_SHAPE;  // beyond the scratch array's capacity
    if (p != p) return PP_ERR_INVALID_ARG;
    if (!x || !y || !Wr || !Wu || !Wd || (d->act == PP_ACT_SWIGLU && !Wg)) return PP_ERR_INVALID_ARG;
    if (!aligned16(x) || !aligned16(y) || !aligned16(Wr) || !aligned16(Wu) || !aligned16(Wd) ||
        (d->act == PP_ACT_SWIGLU && !aligned16(Wg)))
        return PP_ERR_ALIGN;
    if (sel) {
        if (!sel->ids || !sel->counts || !sel->gates) return PP_ERR_INVALID_ARG;
        if (!aligned16(sel->ids) || !aligned16(sel->counts) || !aligned16(sel->gates) ||
            (sel->logits && !aligned16(sel->logits)))
            return PP_ERR_ALIGN;
    }
    return PP_OK;
}

bool encode_down_map(const pp_desc& d, const void* Wd, int rows, CUtensorMap* map) {
    auto enc = pp::tensor_map_encoder();
    if (!enc) return false;
    const bool bf = d.dtype == PP_BF16;
    const cuuint64_t dims[2] = {(cuuint64_t)d.d_ff, (cuuint64_t)d.d_model};
    const cuuint64_t strides[1] = {(cuuint64_t)d.d_ff * (bf ? 2 : 4)};
    const cuuint32_t box[2] = {(cuuint32_t)pp::kDExpert, (cuuint32_t)rows};
    const cuuint32_t estr[2] = {1, 1};
    return enc(map, bf ? CU_TENSOR_MAP_DATA_TYPE_BFLOAT16 : CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 2,
               const_cast<void*>(Wd), dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
               CU_TENSOR_MAP_SWIZZLE_NONE,
               bf ? CU_TENSOR_MAP_L2_PROMOTION_L2_128B : CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

}  // namespace

extern "C" pp_status pp_layer_noalloc(const pp_desc* desc, const void* x, int T, const void* W_r,
                                      const void* W_gate, const void* W_up, const void* W_down, float p,
                                      const pp_selection* sel_out, void* y, uint32_t* status_out, void* stream) {
    const pp_status chk = check_args(desc, T, x, W_r, W_gate, W_up, W_down, p, sel_out, y);
    if (chk != PP_OK) return chk;
    DevState* ds = nullptr;
    const pp_status st0 = device_setup(&ds);
    if (st0 != PP_OK) return st0;
    if (ds->cc_major != 10 || ds->cc_minor != 3) return PP_ERR_UNSUPPORTED;
    if (T == 0) return PP_OK;
    const cudaStream_t st = static_cast<cudaStream_t>(stream);
    const pp_desc& d = *desc;

    // The largest token count one fused launch takes for this shape (pp_layer
    // does the same): fp32 rows of a wide model may fit shared memory only
    // one token at a time.  T is then run in slices of that many tokens.
    int TS = 1;
    while (TS < T) TS <<= 1;
    pp::DecodePlan plan;
    for (;; TS >>= 1) {
        if (TS < 1) return PP_ERR_SHAPE;
        const pp::DecodePlanIn in{d.dtype, d.d_model, d.n_experts, TS, ds->sms, d.act == PP_ACT_SWIGLU,
                                  ds->smem_optin - pp::kDecodeStaticSmemReserve};
        if (pp::decode_plan(in, &plan)) break;
    }

    pp::DecodeArgs a;
    std::memset(&a, 0, sizeof a);
    if (!encode_down_map(d, W_down, plan.R6, &a.tmap_down)) return PP_ERR_CUDA;
    unsigned char* scratch = ds->scratch;
    pp::Control* ctl = reinterpret_cast<pp::Control*>(scratch);
    a.Wr = W_r;
    a.Wg = W_gate;
    a.Wu = W_up;
    a.tlog = reinterpret_cast<unsigned long long*>(scratch + kCtlBytes);
    a.th = reinterpret_cast<unsigned long long*>(scratch + kCtlBytes + kLogitBytes);
    a.epochs = ctl->epoch;
    a.status = &ctl->status;
    a.timeout_ns = kTimeoutNs;
    a.d = d.d_model;
    a.E = d.n_experts;
    a.act = d.act;
    a.gate = d.gate;
    a.rule = d.rule;
    a.p = pp::rule_kernel_param(d.rule, p, d.n_experts);
    a.do_route = 1;
    a.do_ffn = 1;
    a.R6 = plan.R6;
    a.NS4 = plan.NS4;
    a.ded6 = plan.ded6;
    a.slots6 = plan.slots6;
    a.hch = plan.hch;
    a.off_x = plan.off_x;
    a.off_gw = plan.off_gw;
    a.off_mask = plan.off_mask;
    a.off_ulist = plan.off_ulist;
    a.off_red = plan.off_red;
    a.off_red6 = plan.off_red6;
    a.off_ring6 = plan.off_ring6;
    a.off_ring4 = plan.off_ring4;

    // The status word starts at zero for every call.  The launch counts and the tagged words carry over from call to
    // call (zero at load time): a launch only accepts words tagged by itself.
    if (cudaMemsetAsync(&ctl->status, 0, sizeof(unsigned), st) != cudaSuccess) return PP_ERR_CUDA;
    const size_t esz = d.dtype == PP_BF16 ? 2 : 4;
    const size_t E = (size_t)d.n_experts;
    for (int t0 = 0; t0 < T; t0 += TS) {
        const int n = T - t0 < TS ? T - t0 : TS;  // the kernel instance for TS tokens takes any n <= TS
        a.T = n;
        a.x = static_cast<const char*>(x) + (size_t)t0 * d.d_model * esz;
        a.y = static_cast<char*>(y) + (size_t)t0 * d.d_model * esz;
        if (sel_out) {
            a.sel_ids = sel_out->ids + (size_t)t0 * E;
            a.sel_counts = sel_out->counts + t0;
            a.sel_gates = sel_out->gates + (size_t)t0 * E;
            a.sel_logits = sel_out->logits ? sel_out->logits + (size_t)t0 * E : nullptr;
        }
        if (pp::decode_launch(a, plan, d.dtype, TS, ds->sms, st) != cudaSuccess) return PP_ERR_CUDA;
    }
    if (status_out &&
        cudaMemcpyAsync(status_out, &ctl->status, sizeof(uint32_t), cudaMemcpyDeviceToDevice, st) != cudaSuccess)
        return PP_ERR_CUDA;
    return PP_OK;
}
