// C ABI of libprunepath: argument checks, workspace layout and dispatch to
// the kernels.  Everything is enqueued on the caller's stream; nothing here
// allocates device memory or synchronises (except pp_get_device_status).
#include <cmath>
#include <cstring>
#include <mutex>

#include <cudaTypedefs.h>

#include "pp_common.cuh"
#include "pp_kernels.h"

namespace pp {
namespace {

constexpr uint64_t kDefaultTimeoutNs = 2000000000ull;  // bounded waits give up after 2 s

struct DeviceInfo {
    int sms = 0, cc_major = 0, cc_minor = 0;
    size_t smem_optin = 0;
    bool ok = false;
};

DeviceInfo device_info() {
    static std::mutex mu;
    static DeviceInfo cache[64];
    static bool have[64] = {};
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return DeviceInfo{};
    std::lock_guard<std::mutex> lock(mu);
    if (!have[dev]) {
        DeviceInfo d;
        int v = 0;
        bool ok = cudaDeviceGetAttribute(&d.sms, cudaDevAttrMultiProcessorCount, dev) == cudaSuccess;
        ok = ok && cudaDeviceGetAttribute(&d.cc_major, cudaDevAttrComputeCapabilityMajor, dev) == cudaSuccess;
        ok = ok && cudaDeviceGetAttribute(&d.cc_minor, cudaDevAttrComputeCapabilityMinor, dev) == cudaSuccess;
        ok = ok && cudaDeviceGetAttribute(&v, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev) == cudaSuccess;
        d.smem_optin = (size_t)v;
        d.ok = ok;
        cache[dev] = d;
        have[dev] = true;
    }
    return cache[dev];
}

size_t align256(size_t v) { return (v + 255) & ~(size_t)255; }

// Token counts above this use the tensor-core grouped path (bf16 only).
constexpr int kGroupedMinT = 5;

bool use_grouped(const pp_desc& d, int T) { return d.dtype == PP_BF16 && T >= kGroupedMinT; }

// Workspace layout for calls with up to T tokens.
struct Layout {
    size_t logits, ids, counts, gates, tlog, th, stats;
    // grouped path
    size_t part, bits, gexp, invpos, wcnt, blkcnt, blkbase, offsets, n_items, items, perm_token, perm_gate, H, Y,
        yacc, overflow;
    size_t total;
};

Layout layout(const pp_desc& d, int T) {
    const size_t E = (size_t)d.n_experts, Tn = (size_t)(T > 0 ? T : 1);
    Layout L{};
    size_t off = sizeof(Control);
    auto take = [&](size_t bytes) {
        const size_t at = off;
        off = align256(off + bytes);
        return at;
    };
    L.logits = take(Tn * E * 4);
    L.ids = take(Tn * E * 4);
    L.counts = take(Tn * 4);
    L.gates = take(Tn * E * 4);
    // tagged exchange words of the fused decode kernel (up to 8 tokens a launch)
    L.tlog = take(8 * E * 8);
    L.th = take(E * 8 * kDExpert * 8);
    L.stats = take((size_t)router_stats_blocks((int)Tn) * (E + 2) * 8);
    if (use_grouped(d, T)) {
        const GroupedPlan g = grouped_plan(T, d.d_model, d.n_experts, 152);
        L.part = take((size_t)g.nsplit * Tn * E * 4);
        L.bits = take(Tn * 8 * 4);
        L.gexp = take(Tn * E * 4);
        L.invpos = take(Tn * E * 4);
        const size_t nblk = (Tn + 255) / 256;
        L.wcnt = take(nblk * 8 * E * 4);
        L.blkcnt = take(nblk * E * 4);
        L.blkbase = take(nblk * E * 4);
        L.offsets = take((E + 1) * 4);
        L.n_items = take(16);
        L.items = take((size_t)g.max_items * 16);
        L.perm_token = take((size_t)g.nnz_max * 4);
        L.perm_gate = take((size_t)g.nnz_max * 4);
        L.H = take(((size_t)g.nnz_max + 128) * kDExpert * 2);
        L.Y = take((size_t)g.ycap * d.d_model * 2);
        L.yacc = take(Tn * (size_t)d.d_model * 4);
        L.overflow = take(16);
    }
    L.total = off;
    return L;
}

bool aligned16(const void* p) { return ((uintptr_t)p & 15u) == 0; }

pp_status check_desc(const pp_desc* d) {
    if (!d) return PP_ERR_INVALID_ARG;
    if (d->dtype != PP_F32 && d->dtype != PP_BF16) return PP_ERR_DTYPE;
    if (d->act < PP_ACT_RELU || d->act > PP_ACT_SWIGLU) return PP_ERR_INVALID_ARG;
    if (d->gate != PP_GATE_SIGMOID && d->gate != PP_GATE_NONE) return PP_ERR_INVALID_ARG;
    if (!rule_known(d->rule)) return PP_ERR_INVALID_ARG;
    if (d->d_expert != kDExpert) return PP_ERR_SHAPE;
    if (d->n_experts < 1 || d->n_experts > kMaxExperts) return PP_ERR_SHAPE;
    if ((long long)d->d_ff != (long long)d->n_experts * kDExpert) return PP_ERR_SHAPE;
    const int vec = d->dtype == PP_BF16 ? 8 : 4;
    if (d->d_model < 64 || d->d_model > kMaxD || d->d_model % vec != 0) return PP_ERR_SHAPE;
    return PP_OK;
}

pp_status check_T(const pp_desc* d, int T) {
    if (T < 0) return PP_ERR_SHAPE;
    if ((long long)T * d->n_experts > (1ll << 31) - 1 || (long long)T * d->d_model > (1ll << 31) - 1)
        return PP_ERR_SHAPE;
    return PP_OK;
}

pp_status check_ws(const pp_desc* d, int T, void* ws, size_t ws_bytes) {
    if (!ws || ((uintptr_t)ws & 255u) != 0) return PP_ERR_WORKSPACE;
    if (ws_bytes < layout(*d, T).total) return PP_ERR_WORKSPACE;
    return PP_OK;
}

pp_status check_device() {
    const DeviceInfo di = device_info();
    if (!di.ok) return PP_ERR_CUDA;
    if (di.cc_major != 10 || di.cc_minor != 3) return PP_ERR_UNSUPPORTED;
    return PP_OK;
}

pp_status check_sel(const pp_selection* s) {
    if (!s || !s->ids || !s->counts || !s->gates) return PP_ERR_INVALID_ARG;
    if (!aligned16(s->ids) || !aligned16(s->counts) || !aligned16(s->gates)) return PP_ERR_ALIGN;
    if (s->logits && !aligned16(s->logits)) return PP_ERR_ALIGN;
    return PP_OK;
}

pp_status check_weights(const pp_desc* d, const void* Wg, const void* Wu, const void* Wd) {
    if (!Wu || !Wd) return PP_ERR_INVALID_ARG;
    if (d->act == PP_ACT_SWIGLU && !Wg) return PP_ERR_INVALID_ARG;
    if (!aligned16(Wu) || !aligned16(Wd) || (d->act == PP_ACT_SWIGLU && !aligned16(Wg))) return PP_ERR_ALIGN;
    return PP_OK;
}

pp_status cuda_status(cudaError_t e) { return e == cudaSuccess ? PP_OK : PP_ERR_CUDA; }

#define PP_TRY(expr)                        \
    do {                                    \
        const pp_status _s = (expr);        \
        if (_s != PP_OK) return _s;         \
    } while (0)

struct Ws {
    Control* ctrl;
    float* logits;
    int32_t* ids;
    int32_t* counts;
    float* gates;
    unsigned long long* tlog;
    unsigned long long* th;
};

Ws ws_views(const pp_desc& d, int T, void* ws) {
    const Layout L = layout(d, T);
    char* b = static_cast<char*>(ws);
    return Ws{reinterpret_cast<Control*>(b), reinterpret_cast<float*>(b + L.logits),
              reinterpret_cast<int32_t*>(b + L.ids), reinterpret_cast<int32_t*>(b + L.counts),
              reinterpret_cast<float*>(b + L.gates), reinterpret_cast<unsigned long long*>(b + L.tlog),
              reinterpret_cast<unsigned long long*>(b + L.th)};
}

bool make_down_map(const pp_desc& d, const void* Wd, int R6, CUtensorMap* map) {
    auto enc = tensor_map_encoder();
    if (!enc) return false;
    const bool bf = d.dtype == PP_BF16;
    const cuuint64_t dims[2] = {(cuuint64_t)d.d_ff, (cuuint64_t)d.d_model};
    const cuuint64_t strides[1] = {(cuuint64_t)d.d_ff * (bf ? 2 : 4)};
    const cuuint32_t box[2] = {(cuuint32_t)kDExpert, (cuuint32_t)R6};
    const cuuint32_t estr[2] = {1, 1};
    // 128-byte L2 fills for bf16: the next 128 bytes of a row belong to the
    // neighbouring expert, which is usually not selected
    const CUresult r = enc(map, bf ? CU_TENSOR_MAP_DATA_TYPE_BFLOAT16 : CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 2,
                           const_cast<void*>(Wd), dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                           CU_TENSOR_MAP_SWIZZLE_NONE,
                           bf ? CU_TENSOR_MAP_L2_PROMOTION_L2_128B : CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                           CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS;
}

DecodePlanIn plan_in(const pp_desc& d, int TS, bool chain = false) {
    const DeviceInfo di = device_info();
    return DecodePlanIn{d.dtype, d.d_model, d.n_experts, TS, di.sms, d.act == PP_ACT_SWIGLU,
                        di.smem_optin - kDecodeStaticSmemReserve, chain};
}

// The chained step's extra inputs (pp_layer_chained); NULL for a plain layer.
struct Chain {
    const void* y_prev;
    const void* gamma;
    void* x_out;
    float eps;
};

// Largest token count one fused decode launch takes for this shape (0: none).
int decode_ts_limit(const pp_desc& d) {
    for (int ts = decode_max_ts(d.dtype); ts >= 1; ts >>= 1) {
        DecodePlan plan;
        if (decode_plan(plan_in(d, ts), &plan)) return ts;
    }
    return 0;
}

GroupedArgs grouped_args(const pp_desc& d, int T, void* ws, const void* x, const void* Wr, const void* Wg,
                         const void* Wu, const void* Wd, float p, const pp_selection& sel, void* y) {
    const Layout L = layout(d, T);
    char* b = static_cast<char*>(ws);
    GroupedArgs a{};
    a.plan = grouped_plan(T, d.d_model, d.n_experts, 152);
    a.x = x;
    a.Wr = Wr;
    a.Wg = Wg;
    a.Wu = Wu;
    a.Wd = Wd;
    a.y = y;
    a.T = T;
    a.d = d.d_model;
    a.E = d.n_experts;
    a.act = d.act;
    a.gate = d.gate;
    a.rule = d.rule;
    a.p = p;
    a.ids = sel.ids;
    a.counts = sel.counts;
    a.gates = sel.gates;
    a.logits_out = sel.logits;
    a.part = reinterpret_cast<float*>(b + L.part);
    a.bits = reinterpret_cast<uint32_t*>(b + L.bits);
    a.gexp = reinterpret_cast<float*>(b + L.gexp);
    a.invpos = reinterpret_cast<int*>(b + L.invpos);
    a.wcnt = reinterpret_cast<int*>(b + L.wcnt);
    a.blkcnt = reinterpret_cast<int*>(b + L.blkcnt);
    a.blkbase = reinterpret_cast<int*>(b + L.blkbase);
    a.offsets = reinterpret_cast<int*>(b + L.offsets);
    a.n_items = reinterpret_cast<int*>(b + L.n_items);
    a.items = b + L.items;
    a.perm_token = reinterpret_cast<int*>(b + L.perm_token);
    a.perm_gate = reinterpret_cast<float*>(b + L.perm_gate);
    a.H = reinterpret_cast<__nv_bfloat16*>(b + L.H);
    a.Y = reinterpret_cast<__nv_bfloat16*>(b + L.Y);
    a.yacc = reinterpret_cast<float*>(b + L.yacc);
    a.overflow = reinterpret_cast<int*>(b + L.overflow);
    a.status = &reinterpret_cast<Control*>(b)->status;
    a.timeout_ns = kDefaultTimeoutNs;
    return a;
}

// One launch of the fused decode kernel over tokens [t0, t0 + n).
pp_status decode_call(const pp_desc& d, const void* x, int t0, int n, const void* Wr, const void* Wg,
                      const void* Wu, const void* Wd, float p, const pp_selection* sel, bool do_route,
                      bool do_ffn, void* y, const Ws& w, cudaStream_t st, const Chain* chain = nullptr,
                      unsigned long long* tline = nullptr) {
    const DeviceInfo di = device_info();
    int TS = 1;
    while (TS < n) TS <<= 1;
    if (TS > decode_max_ts(d.dtype)) return PP_ERR_SHAPE;
    DecodePlan plan;
    if (!decode_plan(plan_in(d, TS, chain != nullptr), &plan)) return PP_ERR_SHAPE;
    DecodeArgs a;
    std::memset(&a, 0, sizeof a);
    const size_t esz = d.dtype == PP_BF16 ? 2 : 4;
    if (do_ffn && !make_down_map(d, Wd, plan.R6, &a.tmap_down)) return PP_ERR_CUDA;
    const size_t E = (size_t)d.n_experts;
    a.x = static_cast<const char*>(x) + (size_t)t0 * d.d_model * esz;
    a.Wr = Wr;
    a.Wg = Wg;
    a.Wu = Wu;
    a.y = y ? static_cast<char*>(y) + (size_t)t0 * d.d_model * esz : nullptr;
    if (sel) {
        a.sel_ids = sel->ids + (size_t)t0 * E;
        a.sel_counts = sel->counts + t0;
        a.sel_gates = sel->gates + (size_t)t0 * E;
        a.sel_logits = sel->logits ? sel->logits + (size_t)t0 * E : nullptr;
    }
    a.tlog = w.tlog;
    a.th = w.th;
    a.epochs = w.ctrl->epoch;
    a.status = &w.ctrl->status;
    a.timeout_ns = kDefaultTimeoutNs;
    a.T = n;
    a.d = d.d_model;
    a.E = d.n_experts;
    a.act = d.act;
    a.gate = d.gate;
    a.rule = d.rule;
    a.p = p;
    a.do_route = do_route ? 1 : 0;
    a.do_ffn = do_ffn ? 1 : 0;
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
    a.off_chain = plan.off_chain;
    if (chain) {
        const size_t esz = d.dtype == PP_BF16 ? 2 : 4;
        a.chain = 1;
        a.y_prev = chain->y_prev ? static_cast<const char*>(chain->y_prev) + (size_t)t0 * d.d_model * esz : nullptr;
        a.gamma = chain->gamma;
        a.x_out = static_cast<char*>(chain->x_out) + (size_t)t0 * d.d_model * esz;
        a.eps = chain->eps;
    }
    a.tline = tline;
    return cuda_status(decode_launch(a, plan, d.dtype, TS, di.sms, st));
}

}  // namespace

float rule_kernel_param(int rule, float p, int E) {
    if (rule == PP_SEL_TOPK) {
        // k = floor(p) clamped to [1, E]; exact in fp32 since E <= 256
        if (!(p >= 1.0f)) return 1.0f;
        return p >= (float)E ? (float)E : std::floor(p);
    }
    if (rule == PP_SEL_LTE) {
        // Eq. (lte_hard_set): sigmoid(g) > delta  <=>  g > t = ln(delta / (1 - delta));
        // the bound is the smallest float whose value exceeds t
        if (!(p > 0.0f)) return -INFINITY;
        if (p >= 1.0f) return INFINITY;
        const double t = std::log((double)p) - std::log1p(-(double)p);
        float f = (float)t;
        while ((double)f <= t) f = std::nextafter(f, INFINITY);
        while ((double)std::nextafter(f, -INFINITY) > t) f = std::nextafter(f, -INFINITY);
        return f;
    }
    return p;
}

TensorMapEncodeFn tensor_map_encoder() {
    static TensorMapEncodeFn fn = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        void* p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<TensorMapEncodeFn>(p);
    });
    return fn;
}

}  // namespace pp

using namespace pp;

extern "C" {

size_t pp_workspace_size(const pp_desc* desc, int T) {
    if (check_desc(desc) != PP_OK || T < 0) return 0;
    return layout(*desc, T).total;
}

pp_status pp_workspace_init(void* ws, size_t ws_bytes, void* stream) {
    if (!ws || ((uintptr_t)ws & 255u) != 0 || ws_bytes < sizeof(Control)) return PP_ERR_WORKSPACE;
    return cuda_status(cudaMemsetAsync(ws, 0, ws_bytes, static_cast<cudaStream_t>(stream)));
}

pp_status pp_select(const pp_desc* desc, const float* logits, int T, float p, const pp_selection* out,
                    void* ws, size_t ws_bytes, void* stream) {
    PP_TRY(check_desc(desc));
    PP_TRY(check_T(desc, T));
    if (std::isnan(p)) return PP_ERR_INVALID_ARG;
    PP_TRY(check_sel(out));
    if (!logits) return PP_ERR_INVALID_ARG;
    if (!aligned16(logits)) return PP_ERR_ALIGN;
    PP_TRY(check_ws(desc, T, ws, ws_bytes));
    PP_TRY(check_device());
    if (T == 0) return PP_OK;
    const Ws w = ws_views(*desc, T, ws);
    const float kp = rule_kernel_param(desc->rule, p, desc->n_experts);
    return cuda_status(select_launch(logits, T, desc->n_experts, kp, desc->rule, desc->gate, out->ids,
                                     out->counts, out->gates, &w.ctrl->status,
                                     static_cast<cudaStream_t>(stream)));
}

pp_status pp_route(const pp_desc* desc, const void* x, int T, const void* W_r, float p,
                   const pp_selection* out, void* ws, size_t ws_bytes, void* stream) {
    PP_TRY(check_desc(desc));
    PP_TRY(check_T(desc, T));
    if (std::isnan(p)) return PP_ERR_INVALID_ARG;
    PP_TRY(check_sel(out));
    if (!x || !W_r) return PP_ERR_INVALID_ARG;
    if (!aligned16(x) || !aligned16(W_r)) return PP_ERR_ALIGN;
    PP_TRY(check_ws(desc, T, ws, ws_bytes));
    PP_TRY(check_device());
    if (T == 0) return PP_OK;
    const cudaStream_t st = static_cast<cudaStream_t>(stream);
    const Ws w = ws_views(*desc, T, ws);
    const float kp = rule_kernel_param(desc->rule, p, desc->n_experts);
    if (use_grouped(*desc, T)) {
        const GroupedArgs a = grouped_args(*desc, T, ws, x, W_r, nullptr, nullptr, nullptr, kp, *out, nullptr);
        return cuda_status(grouped_route(a, st));
    }
    const int ts = decode_ts_limit(*desc);
    if (ts == 0) return PP_ERR_SHAPE;
    if (T <= ts)
        return decode_call(*desc, x, 0, T, W_r, nullptr, nullptr, nullptr, kp, out, true, false, nullptr, w, st);
    float* lg = out->logits ? out->logits : w.logits;
    PP_TRY(cuda_status(router_launch(desc->dtype, x, T, desc->d_model, W_r, desc->n_experts, lg, st)));
    return cuda_status(select_launch(lg, T, desc->n_experts, kp, desc->rule, desc->gate, out->ids, out->counts,
                                     out->gates, &w.ctrl->status, st));
}

pp_status pp_sparse_ffn(const pp_desc* desc, const void* x, int T, const void* W_gate, const void* W_up,
                        const void* W_down, const pp_selection* sel, void* y, void* ws, size_t ws_bytes,
                        void* stream) {
    PP_TRY(check_desc(desc));
    PP_TRY(check_T(desc, T));
    PP_TRY(check_sel(sel));
    if (!x || !y) return PP_ERR_INVALID_ARG;
    if (!aligned16(x) || !aligned16(y)) return PP_ERR_ALIGN;
    PP_TRY(check_weights(desc, W_gate, W_up, W_down));
    PP_TRY(check_ws(desc, T, ws, ws_bytes));
    PP_TRY(check_device());
    if (T == 0) return PP_OK;
    const cudaStream_t st = static_cast<cudaStream_t>(stream);
    const Ws w = ws_views(*desc, T, ws);
    if (use_grouped(*desc, T)) {
        const GroupedArgs a = grouped_args(*desc, T, ws, x, nullptr, W_gate, W_up, W_down, 0.0f, *sel, y);
        return cuda_status(grouped_ffn(a, device_info().sms, st));
    }
    const int ts = decode_ts_limit(*desc);
    if (ts == 0) return PP_ERR_SHAPE;
    for (int t0 = 0; t0 < T; t0 += ts) {
        const int n = std::min(ts, T - t0);
        PP_TRY(decode_call(*desc, x, t0, n, nullptr, W_gate, W_up, W_down, 0.0f, sel, false, true, y, w, st));
    }
    return PP_OK;
}

pp_status pp_layer(const pp_desc* desc, const void* x, int T, const void* W_r, const void* W_gate,
                   const void* W_up, const void* W_down, float p, const pp_selection* sel_out, void* y,
                   void* ws, size_t ws_bytes, void* stream) {
    PP_TRY(check_desc(desc));
    PP_TRY(check_T(desc, T));
    if (std::isnan(p)) return PP_ERR_INVALID_ARG;
    if (sel_out) PP_TRY(check_sel(sel_out));
    if (!x || !y || !W_r) return PP_ERR_INVALID_ARG;
    if (!aligned16(x) || !aligned16(y) || !aligned16(W_r)) return PP_ERR_ALIGN;
    PP_TRY(check_weights(desc, W_gate, W_up, W_down));
    PP_TRY(check_ws(desc, T, ws, ws_bytes));
    PP_TRY(check_device());
    if (T == 0) return PP_OK;
    const cudaStream_t st = static_cast<cudaStream_t>(stream);
    const Ws w = ws_views(*desc, T, ws);
    pp_selection s = sel_out ? *sel_out : pp_selection{w.ids, w.counts, w.gates, nullptr};
    const float kp = rule_kernel_param(desc->rule, p, desc->n_experts);
    if (use_grouped(*desc, T)) {
        const GroupedArgs a = grouped_args(*desc, T, ws, x, W_r, W_gate, W_up, W_down, kp, s, y);
        PP_TRY(cuda_status(grouped_route(a, st)));
        return cuda_status(grouped_ffn(a, device_info().sms, st));
    }
    const int ts = decode_ts_limit(*desc);
    if (ts == 0) return PP_ERR_SHAPE;
    if (T <= ts)
        return decode_call(*desc, x, 0, T, W_r, W_gate, W_up, W_down, kp, sel_out, true, true, y, w, st);
    float* lg = s.logits ? s.logits : w.logits;
    PP_TRY(cuda_status(router_launch(desc->dtype, x, T, desc->d_model, W_r, desc->n_experts, lg, st)));
    PP_TRY(cuda_status(select_launch(lg, T, desc->n_experts, kp, desc->rule, desc->gate, s.ids, s.counts, s.gates,
                                     &w.ctrl->status, st)));
    for (int t0 = 0; t0 < T; t0 += ts) {
        const int n = std::min(ts, T - t0);
        PP_TRY(decode_call(*desc, x, t0, n, nullptr, W_gate, W_up, W_down, 0.0f, &s, false, true, y, w, st));
    }
    return PP_OK;
}

pp_status pp_layer_chained(const pp_desc* desc, const void* x_prev, const void* y_prev, const void* gamma, float eps,
                           int T, const void* W_r, const void* W_gate, const void* W_up, const void* W_down, float p,
                           const pp_selection* sel_out, void* x, void* y, void* ws, size_t ws_bytes, void* stream) {
    PP_TRY(check_desc(desc));
    PP_TRY(check_T(desc, T));
    if (std::isnan(p) || !(eps >= 0.0f)) return PP_ERR_INVALID_ARG;
    if (sel_out) PP_TRY(check_sel(sel_out));
    if (!x_prev || !x || !y || !W_r) return PP_ERR_INVALID_ARG;
    if (!aligned16(x_prev) || !aligned16(x) || !aligned16(y) || !aligned16(W_r) || (y_prev && !aligned16(y_prev)) ||
        (gamma && !aligned16(gamma)))
        return PP_ERR_ALIGN;
    // x and y are written while other CTAs may still read x_prev / y_prev
    const size_t rows = (size_t)T * desc->d_model * (desc->dtype == PP_BF16 ? 2 : 4);
    auto overlap = [rows](const void* a, const void* b) {
        const char* pa = static_cast<const char*>(a);
        const char* pb = static_cast<const char*>(b);
        return a && b && pa < pb + rows && pb < pa + rows;
    };
    if (overlap(x, x_prev) || overlap(x, y_prev) || overlap(y, x_prev) || overlap(y, y_prev) || overlap(x, y))
        return PP_ERR_INVALID_ARG;
    PP_TRY(check_weights(desc, W_gate, W_up, W_down));
    PP_TRY(check_ws(desc, T, ws, ws_bytes));
    PP_TRY(check_device());
    if (T == 0) return PP_OK;
    const cudaStream_t st = static_cast<cudaStream_t>(stream);
    const Ws w = ws_views(*desc, T, ws);
    // fused: the decode kernel forms x in its prologue
    if (!use_grouped(*desc, T)) {
        const int ts = decode_ts_limit(*desc);
        DecodePlan plan;
        int TS = 1;
        while (TS < T) TS <<= 1;
        if (ts > 0 && T <= ts && decode_plan(plan_in(*desc, TS, true), &plan)) {
            const float kp = rule_kernel_param(desc->rule, p, desc->n_experts);
            const Chain c{y_prev, gamma, x, eps};
            return decode_call(*desc, x_prev, 0, T, W_r, W_gate, W_up, W_down, kp, sel_out, true, true, y, w, st, &c);
        }
    }
    // otherwise x first, then the layer on it
    PP_TRY(cuda_status(rmsnorm_residual_launch(desc->dtype, x_prev, y_prev, gamma, eps, T, desc->d_model, x, st)));
    return pp_layer(desc, x, T, W_r, W_gate, W_up, W_down, p, sel_out, y, ws, ws_bytes, stream);
}

pp_status pp_sparsity_stats(const int32_t* counts, int T, int n_experts, uint64_t* acc, void* stream) {
    if (!counts || !acc || T < 0 || n_experts < 1 || n_experts > kMaxExperts) return PP_ERR_INVALID_ARG;
    if (((uintptr_t)counts & 3u) || ((uintptr_t)acc & 7u)) return PP_ERR_ALIGN;
    PP_TRY(check_device());
    return cuda_status(stats_launch(counts, T, n_experts, acc, static_cast<cudaStream_t>(stream)));
}

pp_status pp_router_stats(const pp_desc* desc, const float* logits, int T, float eps, double* out, void* ws,
                          size_t ws_bytes, void* stream) {
    PP_TRY(check_desc(desc));
    PP_TRY(check_T(desc, T));
    if (T < 1) return PP_ERR_SHAPE;
    if (std::isnan(eps) || !logits || !out) return PP_ERR_INVALID_ARG;
    if (!aligned16(logits) || ((uintptr_t)out & 7u)) return PP_ERR_ALIGN;
    PP_TRY(check_ws(desc, T, ws, ws_bytes));
    PP_TRY(check_device());
    char* b = static_cast<char*>(ws);
    float* part = reinterpret_cast<float*>(b + layout(*desc, T).stats);
    return cuda_status(router_stats_launch(logits, T, desc->n_experts, eps, part, out,
                                           &reinterpret_cast<Control*>(b)->status,
                                           static_cast<cudaStream_t>(stream)));
}

pp_status pp_moefy_cluster(const pp_desc* desc, const void* W_gate, const void* W_up, const int32_t* init,
                           int max_iter, int32_t* perm, int32_t* labels, int* iters, double* objective) {
    PP_TRY(check_desc(desc));
    const bool gated = desc->act == PP_ACT_SWIGLU;
    if (!W_up || !init || !perm || (gated && !W_gate) || max_iter < 1) return PP_ERR_INVALID_ARG;
    const int E = desc->n_experts, dff = desc->d_ff;
    uint32_t seen[kMaxExperts * kDExpert / 32] = {};  // d_ff <= 256 * 64 bits
    for (int h = 0; h < E; ++h) {
        const int v = init[h];
        if (v < 0 || v >= dff || (seen[v >> 5] >> (v & 31) & 1u)) return PP_ERR_INVALID_ARG;
        seen[v >> 5] |= 1u << (v & 31);
    }
    return moefy_cluster_host(desc->dtype, gated ? W_gate : nullptr, W_up, dff, desc->d_model, E, init, max_iter,
                              labels, perm, iters, objective);
}

pp_status pp_moefy_permute(const pp_desc* desc, const int32_t* perm, const void* W_gate, const void* W_up,
                           const void* W_down, void* W_gate_out, void* W_up_out, void* W_down_out, void* ws,
                           size_t ws_bytes, void* stream) {
    PP_TRY(check_desc(desc));
    const bool gated = desc->act == PP_ACT_SWIGLU;
    if (!perm || !W_up_out || !W_down_out || (gated && !W_gate_out)) return PP_ERR_INVALID_ARG;
    PP_TRY(check_weights(desc, gated ? W_gate : nullptr, W_up, W_down));
    if (!aligned16(perm) || !aligned16(W_up_out) || !aligned16(W_down_out) || (gated && !aligned16(W_gate_out)))
        return PP_ERR_ALIGN;
    const size_t mat = (size_t)desc->d_ff * desc->d_model * (desc->dtype == PP_BF16 ? 2 : 4);
    const char* in[3] = {static_cast<const char*>(gated ? W_gate : nullptr), static_cast<const char*>(W_up),
                         static_cast<const char*>(W_down)};
    const char* out[3] = {static_cast<const char*>(gated ? W_gate_out : nullptr),
                          static_cast<const char*>(W_up_out), static_cast<const char*>(W_down_out)};
    auto overlap = [mat](const char* a, const char* b) { return a && b && a < b + mat && b < a + mat; };
    for (int i = 0; i < 3; ++i) {
        for (int j = 0; j < 3; ++j) {
            if (overlap(out[i], in[j])) return PP_ERR_INVALID_ARG;
            if (j > i && overlap(out[i], out[j])) return PP_ERR_INVALID_ARG;
        }
        const char* pe = reinterpret_cast<const char*>(perm);
        if (out[i] && out[i] < pe + (size_t)desc->d_ff * 4 && pe < out[i] + mat) return PP_ERR_INVALID_ARG;
    }
    PP_TRY(check_ws(desc, 0, ws, ws_bytes));
    PP_TRY(check_device());
    const DeviceInfo di = device_info();
    return cuda_status(moefy_permute_launch(desc->dtype, perm, gated ? W_gate : nullptr, W_up, W_down,
                                            gated ? W_gate_out : nullptr, W_up_out, W_down_out, desc->d_model,
                                            desc->d_ff, di.sms, &static_cast<Control*>(ws)->status,
                                            static_cast<cudaStream_t>(stream)));
}

pp_status pp_get_device_status(void* ws, void* stream) {
    if (!ws || ((uintptr_t)ws & 255u) != 0) return PP_ERR_WORKSPACE;
    const cudaStream_t st = static_cast<cudaStream_t>(stream);
    unsigned v = 0;
    if (cudaMemcpyAsync(&v, &static_cast<Control*>(ws)->status, sizeof v, cudaMemcpyDeviceToHost, st) !=
        cudaSuccess)
        return PP_ERR_CUDA;
    if (cudaStreamSynchronize(st) != cudaSuccess) return PP_ERR_CUDA;
    return static_cast<pp_status>(v);
}

pp_status pp_debug_decode_timeline(const pp_desc* desc, const void* x, const void* W_r, const void* W_gate,
                                    const void* W_up, const void* W_down, float p, void* y, void* ws, size_t ws_bytes,
                                    uint64_t* stamps, size_t stamps_bytes, void* stream) {
    PP_TRY(check_desc(desc));
    if (desc->dtype != PP_BF16) return PP_ERR_DTYPE;
    if (std::isnan(p)) return PP_ERR_INVALID_ARG;
    if (!x || !y || !W_r || !stamps) return PP_ERR_INVALID_ARG;
    if (!aligned16(x) || !aligned16(y) || !aligned16(W_r) || !aligned16(stamps)) return PP_ERR_ALIGN;
    PP_TRY(check_weights(desc, W_gate, W_up, W_down));
    PP_TRY(check_ws(desc, 1, ws, ws_bytes));
    PP_TRY(check_device());
    if (stamps_bytes < (size_t)kMaxGrid * kDecodeStamps * sizeof(uint64_t)) return PP_ERR_INVALID_ARG;
    if (decode_ts_limit(*desc) < 1) return PP_ERR_SHAPE;
    const cudaStream_t st = static_cast<cudaStream_t>(stream);
    const Ws w = ws_views(*desc, 1, ws);
    const float kp = rule_kernel_param(desc->rule, p, desc->n_experts);
    return decode_call(*desc, x, 0, 1, W_r, W_gate, W_up, W_down, kp, nullptr, true, true, y, w, st, nullptr,
                       reinterpret_cast<unsigned long long*>(stamps));
}

pp_status pp_debug_wait_timeout(void* ws, size_t ws_bytes, long long timeout_ns, void* stream) {
    if (!ws || ((uintptr_t)ws & 255u) != 0 || ws_bytes < sizeof(Control)) return PP_ERR_WORKSPACE;
    if (timeout_ns <= 0 || timeout_ns > 10000000000ll) return PP_ERR_INVALID_ARG;
    PP_TRY(check_device());
    Control* c = static_cast<Control*>(ws);
    return cuda_status(wait_timeout_launch(&c->wait_flag, &c->status, timeout_ns, static_cast<cudaStream_t>(stream)));
}

const char* pp_status_string(pp_status s) {
    switch (s) {
        case PP_OK: return "PP_OK";
        case PP_ERR_INVALID_ARG: return "PP_ERR_INVALID_ARG";
        case PP_ERR_SHAPE: return "PP_ERR_SHAPE";
        case PP_ERR_DTYPE: return "PP_ERR_DTYPE";
        case PP_ERR_ALIGN: return "PP_ERR_ALIGN";
        case PP_ERR_WORKSPACE: return "PP_ERR_WORKSPACE";
        case PP_ERR_CUDA: return "PP_ERR_CUDA";
        case PP_ERR_TIMEOUT: return "PP_ERR_TIMEOUT";
        case PP_ERR_CAPACITY: return "PP_ERR_CAPACITY";
        case PP_ERR_NONFINITE: return "PP_ERR_NONFINITE";
        case PP_ERR_UNSUPPORTED: return "PP_ERR_UNSUPPORTED";
        case PP_ERR_HOST: return "PP_ERR_HOST";
    }
    return "PP_ERR_UNKNOWN";
}

const char* pp_version(void) { return "0.1.0"; }

}  // extern "C"
