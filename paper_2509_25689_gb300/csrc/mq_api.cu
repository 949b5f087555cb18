// C ABI of libmoeq: argument checks, workspace carving, kernel dispatch,
// optional kernel timing.  See include/moeq.h for the contract.
#include <cuda_runtime.h>

#include <cmath>
#include <cstdlib>
#include <cstring>
#include <mutex>
#include <string>
#include <vector>

#include "../../include/moeq.h"
#include "mq_actprep.cuh"
#include "mq_internal.h"

namespace mq {
namespace {

size_t up256(size_t v) { return (v + 255) & ~size_t(255); }

constexpr int32_t kFusedRouteTokens = 256;   // up to this many tokens: one routing CTA

int g_path_mode = -1;        // -1: not yet read from the environment
// automatic path choice: the grouped GEMM from this many tokens on (on the
// V3 layer with mixed formats it is the faster path from about 50 tokens:
// 48 tokens 2.46 ms decode / 2.50 ms GEMM, 56 tokens 2.83 / 2.64 ms)
int32_t g_prefill_threshold = 50;

int path_mode() {
    if (g_path_mode < 0) {
        const char* env = std::getenv("MQ_FORCE_PATH");
        g_path_mode = 0;
        if (env && std::strcmp(env, "decode") == 0) g_path_mode = 1;
        if (env && std::strcmp(env, "prefill") == 0) g_path_mode = 2;
        if (env && std::strcmp(env, "decode_tc") == 0) g_path_mode = 3;
    }
    return g_path_mode;
}

}  // namespace

// the mma.sync decode kernels (k_decode.cu) stream whole 256-element superblocks
bool decode_mma_fits(const Dims& d) { return d.H % 256 == 0 && d.I % 256 == 0; }

namespace {

int check_cfg(const mq_layer_cfg* c) {
    if (!c) return MQ_EINVAL;
    if (c->hidden < 128 || c->hidden % 128 || c->hidden > 32768) return MQ_ESHAPE;
    if (c->inter < 128 || c->inter % 128 || c->inter > 16384) return MQ_ESHAPE;
    if (c->n_experts < 1 || c->n_experts > kMaxExperts) return MQ_ESHAPE;
    if (c->n_groups < 1 || c->n_groups > kMaxGroups || c->n_experts % c->n_groups) return MQ_ESHAPE;
    if (c->topk_group < 1 || c->topk_group > c->n_groups) return MQ_ESHAPE;
    if (c->top_k < 1 || c->top_k > kMaxTopK) return MQ_ESHAPE;
    if (c->top_k > c->topk_group * (c->n_experts / c->n_groups)) return MQ_ESHAPE;
    if (c->has_shared != 0 && c->has_shared != 1) return MQ_EINVAL;
    if (!std::isfinite(c->routed_scale)) return MQ_EINVAL;
    return MQ_OK;
}

Dims dims_of(const mq_layer_cfg* c, int32_t T) {
    Dims d;
    d.H = c->hidden; d.I = c->inter; d.E = c->n_experts; d.G = c->n_groups; d.Gk = c->topk_group;
    d.K = c->top_k; d.T = T; d.has_shared = c->has_shared; d.routed_scale = c->routed_scale;
    d.x_fams = kCodeFams;
    return d;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

// ---- kernel timing -------------------------------------------------------
struct ProfRec { const char* name; cudaEvent_t a, b; };
std::mutex g_prof_mu;
bool g_prof_on = false;
int32_t g_prof_cap = 0;
std::vector<ProfRec> g_prof;

}  // namespace

size_t workspace_plan(const Dims& d, void* base, Work* w) {
    const size_t TK = (size_t)d.T * d.K;
    const size_t A = TK + (size_t)d.T;             // routed assignments + shared-expert rows
    const size_t nsbx = (size_t)(d.H + 255) / 256, nsbi = (size_t)(d.I + 255) / 256;
    size_t at = 0;
    auto take = [&](size_t bytes) { const size_t o = at; at += up256(bytes); return o; };
    const size_t o_z = take((size_t)d.T * d.E * 4);
    const size_t o_idx = take(TK * 4), o_w = take(TK * 4);
    const size_t o_off = take((size_t)(d.E + 1) * 4);
    const size_t o_perm = take(TK * 4), o_inv = take(TK * 4);
    const size_t o_act = take((size_t)(d.E + 2) * 4);
    const size_t o_xq = take((size_t)d.T * kFamSlots * nsbx * 256 * 2);
    const size_t o_xs = take((size_t)d.T * nsbx * kStatFloats * 4);
    const size_t o_hq = take(A * kFamSlots * nsbi * 256 * 2);
    const size_t o_hs = take(A * nsbi * kStatFloats * 4);
    const size_t o_pdn = take(A * d.H * 4);
    const size_t o_plan = take(sizeof(Plan));
    const size_t o_xe = take((size_t)d.T * 4);
    const size_t o_spart = take((size_t)d.T * 4 * d.I * 4);   // shared gate/up K halves (decode)
    const size_t cnt_bytes = decode_counter_bytes(d);
    // work counters, the two routing words, then the error word (zeroed per call)
    const size_t o_cnt = take(cnt_bytes + 12);
    const size_t o_sync = o_cnt + cnt_bytes;
    const size_t o_err = o_sync + 8;
    if (w && base) {
        char* b = static_cast<char*>(base);
        w->z = reinterpret_cast<float*>(b + o_z);
        w->idx = reinterpret_cast<int32_t*>(b + o_idx);
        w->wts = reinterpret_cast<float*>(b + o_w);
        w->offsets = reinterpret_cast<int32_t*>(b + o_off);
        w->perm = reinterpret_cast<int32_t*>(b + o_perm);
        w->inv = reinterpret_cast<int32_t*>(b + o_inv);
        w->active = reinterpret_cast<int32_t*>(b + o_act);
        w->xq = reinterpret_cast<__half*>(b + o_xq);
        w->xs = reinterpret_cast<float*>(b + o_xs);
        w->hq = reinterpret_cast<__half*>(b + o_hq);
        w->hs = reinterpret_cast<float*>(b + o_hs);
        w->pdn = reinterpret_cast<float*>(b + o_pdn);
        w->plan = reinterpret_cast<Plan*>(b + o_plan);
        w->counters = reinterpret_cast<uint32_t*>(b + o_cnt);
        w->counter_bytes = cnt_bytes;
        w->logits_done = reinterpret_cast<uint32_t*>(b + o_sync);
        w->route_ready = reinterpret_cast<uint32_t*>(b + o_sync + 4);
        w->err = reinterpret_cast<uint32_t*>(b + o_err);
        w->xe = reinterpret_cast<int32_t*>(b + o_xe);
        w->spart = reinterpret_cast<float*>(b + o_spart);
        w->x16 = w->xq;   // the prefill path uses these bytes instead of the decode preparation
        w->h16 = w->hq;
        w->zero_words = w->counters;
        w->n_zero = (int)((cnt_bytes + 12) / 4);
    }
    return at;
}

namespace {
constexpr int kMaxSetupDevices = 64;
std::mutex g_setup_mu;
int g_setup_sms[kMaxSetupDevices][kSetupSlots] = {};
}  // namespace

int device_setup(int slot, void (*init)()) {
    int dev = -1;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxSetupDevices || slot < 0 || slot >= kSetupSlots)
        return 0;
    std::lock_guard<std::mutex> lk(g_setup_mu);
    int& sms = g_setup_sms[dev][slot];
    if (sms == 0) {
        int n = 0;
        if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0) return 0;
        if (init) init();
        sms = n;
    }
    return sms;
}

namespace {
std::mutex g_wait_test_mu;
uint64_t g_wait_test_ns = 0;   // armed when non-zero
}  // namespace

bool take_wait_test(uint64_t* wait_ns) {
    std::lock_guard<std::mutex> lk(g_wait_test_mu);
    if (g_wait_test_ns == 0) return false;
    *wait_ns = g_wait_test_ns;
    g_wait_test_ns = 0;
    return true;
}

void prof_begin(const char* name, cudaStream_t s) {
    std::lock_guard<std::mutex> lk(g_prof_mu);
    if (!g_prof_on || (int32_t)g_prof.size() >= g_prof_cap) return;
    ProfRec r{name, nullptr, nullptr};
    cudaEventCreate(&r.a);
    cudaEventCreate(&r.b);
    cudaEventRecord(r.a, s);
    g_prof.push_back(r);
}

void prof_end(cudaStream_t s) {
    std::lock_guard<std::mutex> lk(g_prof_mu);
    if (!g_prof_on || g_prof.empty()) return;
    ProfRec& r = g_prof.back();
    if (r.b) cudaEventRecord(r.b, s);
}

}  // namespace mq

using namespace mq;

extern "C" const char* mq_strerror(int status) {
    switch (status) {
    case MQ_OK: return "ok";
    case MQ_EINVAL: return "invalid argument";
    case MQ_EFORMAT: return "unknown packed format";
    case MQ_EALIGN: return "pointer not 16-byte aligned";
    case MQ_ESHAPE: return "inconsistent layer shape";
    case MQ_EWORKSPACE: return "workspace missing or too small";
    case MQ_ECUDA: return "CUDA error";
    case MQ_EDEVICE: return "device-side check failed";
    case MQ_ERANGE: return "size beyond supported maximum";
    default: return "unknown status";
    }
}

extern "C" int mq_set_path(int mode, int32_t prefill_threshold) {
    if (mode < 0 || mode > 3) return MQ_EINVAL;
    path_mode();
    g_path_mode = mode;
    if (prefill_threshold > 0) g_prefill_threshold = prefill_threshold;
    return MQ_OK;
}

extern "C" size_t moe_quant_workspace_size(const mq_layer_cfg* cfg, int32_t n_tokens) {
    if (check_cfg(cfg) != MQ_OK || n_tokens < 0 || n_tokens > 65536) return 0;
    return workspace_plan(dims_of(cfg, n_tokens), nullptr, nullptr);
}

namespace {

int check_common(const mq_layer_cfg* cfg, int32_t T, const void* x, const float* router_w, const float* bias,
                 void* ws, size_t ws_bytes) {
    const int rc = check_cfg(cfg);
    if (rc != MQ_OK) return rc;
    if (T < 0 || T > 65536) return MQ_ESHAPE;
    if (T > 0 && (!x || !router_w)) return MQ_EINVAL;
    if (T > 0 && (!aligned16(x) || !aligned16(router_w))) return MQ_EALIGN;
    (void)bias;
    const size_t need = workspace_plan(dims_of(cfg, T), nullptr, nullptr);
    if (!ws || ws_bytes < need || (reinterpret_cast<uintptr_t>(ws) & 255u)) return MQ_EWORKSPACE;
    return MQ_OK;
}

// Routing, permutation and the per-call set-up of the expert-FFN path:
// mode 0 = routing only, 1 = decode (prepared tokens + work plan),
// 2 = prefill (fp16 tokens for the grouped GEMM).  Forward calls first clear
// their per-call words.  fuse (decode on the mma.sync kernels): the logits
// kernel's last CTA routes and permutes, and the expert-FFN kernel follows
// it directly, waiting on the published flags.
int run_route(const Dims& d, const void* x, const float* router_w, const float* bias, Work& w,
              cudaStream_t s, int mode, bool fuse = false) {
    const bool fwd = mode != 0;
    if (fwd && launch_zero(w.zero_words, w.n_zero, s) != cudaSuccess) return MQ_ECUDA;
    Plan* plan = mode == 1 ? w.plan : nullptr;
    if (fuse) {
        FusedRoute fr{};
        fr.d = d;
        fr.bias = bias;
        // the expert-FFN kernel reads the plan and the permutation only
        fr.idx = w.idx; fr.wts = w.wts; fr.offsets = nullptr; fr.perm = w.perm; fr.inv = nullptr;
        fr.active = nullptr; fr.plan = plan;
        fr.logits_done = w.logits_done;
        fr.route_ready = w.route_ready;
        if (launch_router_logits(d, static_cast<const uint16_t*>(x), router_w, w.z, w.xq, w.xs, nullptr, w.xe, &fr,
                                 s) != cudaSuccess)
            return MQ_ECUDA;
        return MQ_OK;
    }
    if (launch_router_logits(d, static_cast<const uint16_t*>(x), router_w, w.z, mode == 1 ? w.xq : nullptr, w.xs,
                             mode == 2 ? w.x16 : nullptr, w.xe, nullptr, s) != cudaSuccess)
        return MQ_ECUDA;
    if (d.T <= kFusedRouteTokens) {
        // decode-sized batch: top-k, permutation and work plan in one CTA
        if (launch_route_permute(d, w.z, bias, w.idx, w.wts, w.offsets, w.perm, w.inv, w.active, plan, s) !=
            cudaSuccess)
            return MQ_ECUDA;
        return MQ_OK;
    }
    if (launch_topk(d, w.z, bias, w.idx, w.wts, s) != cudaSuccess) return MQ_ECUDA;
    if (launch_permute(d, w.idx, w.offsets, w.perm, w.inv, w.active, plan, s) != cudaSuccess) return MQ_ECUDA;
    return MQ_OK;
}

}  // namespace

extern "C" int moe_quant_route(const mq_layer_cfg* cfg, int32_t n_tokens, const void* x, const float* router_w,
                               const float* bias, int32_t* topk_idx, float* topk_w, int32_t* offsets,
                               int32_t* perm, int32_t* inv, void* workspace, size_t ws_bytes, void* stream) {
    int rc = check_common(cfg, n_tokens, x, router_w, bias, workspace, ws_bytes);
    if (rc != MQ_OK) return rc;
    if (n_tokens > 0 && (!topk_idx || !topk_w)) return MQ_EINVAL;
    const Dims d = dims_of(cfg, n_tokens);
    Work w;
    workspace_plan(d, workspace, &w);
    w.idx = topk_idx;
    w.wts = topk_w;
    if (offsets) w.offsets = offsets;
    if (perm) w.perm = perm;
    if (inv) w.inv = inv;
    return run_route(d, x, router_w, bias, w, static_cast<cudaStream_t>(stream), 0);
}

extern "C" int moe_quant_forward(const mq_layer_cfg* cfg, int32_t n_tokens, const void* x, const float* router_w,
                                 const float* bias, const mq_expert_table* table, const uint8_t* fmt,
                                 float* out, int32_t* topk_idx, float* topk_w, void* workspace, size_t ws_bytes,
                                 void* stream) {
    int rc = check_common(cfg, n_tokens, x, router_w, bias, workspace, ws_bytes);
    if (rc != MQ_OK) return rc;
    if (!table || !table->experts || !fmt) return MQ_EINVAL;
    if (cfg->has_shared && !table->shared) return MQ_EINVAL;
    if (n_tokens > 0 && !out) return MQ_EINVAL;
    Dims d = dims_of(cfg, n_tokens);
    static thread_local ExpertTab tab;
    const int n = d.E + d.has_shared;
    bool new_fmts = false;   // Q6_K / BF16 tensors: not on the tcgen05 GEMV kernels
    for (int e = 0; e < n; ++e) {
        const mq_expert_weights& ew = e < d.E ? table->experts[e] : *table->shared;
        const void* ps[3] = {ew.gate, ew.up, ew.down};
        for (int j = 0; j < 3; ++j) {
            const int f = fmt[3 * e + j];
            if (!valid_format(f)) return MQ_EFORMAT;
            if (!ps[j]) return MQ_EINVAL;
            if (!aligned16(ps[j])) return MQ_EALIGN;
            tab.p[e][j] = static_cast<const uint8_t*>(ps[j]);
            tab.fmt[e][j] = (uint8_t)f;
            new_fmts |= f == kQ6K || f == kBF16;
            if (f == kBF16 && j < 2) d.x_fams |= kBf16Fams;   // bf16 operands of the tokens
        }
    }
    if (n_tokens == 0) return MQ_OK;
    const cudaStream_t s = static_cast<cudaStream_t>(stream);
    Work w;
    workspace_plan(d, workspace, &w);
    if (topk_idx) w.idx = topk_idx;
    if (topk_w) w.wts = topk_w;
    const int pm = path_mode();
    bool prefill = pm == 2 || (pm == 0 && n_tokens >= g_prefill_threshold);
    const bool tc = !prefill && decode_tc_fits(d) && (pm == 3 || !decode_mma_fits(d));
    if (tc && new_fmts) {
        // the tcgen05 GEMV kernels take Q2_K/Q3_K/Q4_K/Q8_0 only: a forced
        // request is refused, an automatic choice goes to the grouped GEMM
        if (pm == 3) return MQ_EFORMAT;
        prefill = true;
    }
    rc = run_route(d, x, router_w, bias, w, s, prefill ? 2 : 1, !prefill && !tc);
    if (rc != MQ_OK) return rc;
    if (prefill) {
        if (launch_prefill(d, tab, w, out, s) != cudaSuccess) return MQ_ECUDA;
        return MQ_OK;
    }
    const cudaError_t e = tc ? launch_decode_tc(d, tab, w, out, s) : launch_decode_mma(d, tab, w, out, s);
    if (e != cudaSuccess) return MQ_ECUDA;
    return MQ_OK;
}

// ---------------------------------------------------------------------------
// Forward pass that allocates nothing: its scratch is a fixed device array
// owned by this library.  For callers that cannot call cudaMalloc (see
// include/moeq.h).
// ---------------------------------------------------------------------------
namespace {

constexpr size_t kNoAllocScratchBytes = size_t(16) << 20;   // 16 MiB
constexpr int kNoAllocMaxDevices = 64;

// Every device that loads this library holds this array until the process
// exits.  Host code must not pass `g_noalloc_scratch` itself to a kernel: on
// the host the name is only a stand-in for the device symbol, so its device
// address is looked up once per device below.
static __device__ __align__(256) uint8_t g_noalloc_scratch[kNoAllocScratchBytes];

std::mutex g_noalloc_mu;
void* g_noalloc_ptr[kNoAllocMaxDevices] = {};

// Device address of the scratch array on the current device (looked up on
// the first call made with that device current).
int noalloc_scratch(void** out) {
    int dev = -1;
    if (cudaGetDevice(&dev) != cudaSuccess) return MQ_ECUDA;
    if (dev < 0 || dev >= kNoAllocMaxDevices) return MQ_ERANGE;
    std::lock_guard<std::mutex> lk(g_noalloc_mu);
    if (!g_noalloc_ptr[dev]) {
        void* p = nullptr;
        if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess || !p) return MQ_ECUDA;
        g_noalloc_ptr[dev] = p;
    }
    *out = g_noalloc_ptr[dev];
    return MQ_OK;
}

}  // namespace

extern "C" int moe_quant_forward_noalloc(const mq_layer_cfg* cfg, int32_t n_tokens, const void* x,
                                         const float* router_w, const float* bias, const mq_expert_table* table,
                                         const uint8_t* fmt, float* out, int32_t* topk_idx, float* topk_w,
                                         void* stream) {
    const int rc = check_cfg(cfg);
    if (rc != MQ_OK) return rc;
    if (n_tokens < 0 || n_tokens > 65536) return MQ_ESHAPE;
    if (workspace_plan(dims_of(cfg, n_tokens), nullptr, nullptr) > kNoAllocScratchBytes) return MQ_ERANGE;
    void* scratch = nullptr;
    const int sr = noalloc_scratch(&scratch);
    if (sr != MQ_OK) return sr;
    // the forward pass clears the parts of its scratch that must start at zero
    return moe_quant_forward(cfg, n_tokens, x, router_w, bias, table, fmt, out, topk_idx, topk_w, scratch,
                             kNoAllocScratchBytes, stream);
}

namespace {

// Reads the error word of the workspace laid out for (cfg, n_tokens) once the
// stream's work is done.
int read_status(const mq_layer_cfg* cfg, int32_t n_tokens, const void* ws, size_t ws_bytes, uint32_t* err_bits,
                void* stream) {
    const int rc = check_cfg(cfg);
    if (rc != MQ_OK) return rc;
    if (n_tokens < 0 || n_tokens > 65536) return MQ_ESHAPE;
    const Dims d = dims_of(cfg, n_tokens);
    const size_t need = workspace_plan(d, nullptr, nullptr);
    if (!ws || ws_bytes < need || (reinterpret_cast<uintptr_t>(ws) & 255u)) return MQ_EWORKSPACE;
    if (err_bits) *err_bits = 0;
    if (n_tokens == 0) return MQ_OK;   // a call without tokens launches nothing
    Work w;
    workspace_plan(d, const_cast<void*>(ws), &w);
    const cudaStream_t s = static_cast<cudaStream_t>(stream);
    uint32_t v = 0;
    if (cudaMemcpyAsync(&v, w.err, sizeof(v), cudaMemcpyDeviceToHost, s) != cudaSuccess) return MQ_ECUDA;
    if (cudaStreamSynchronize(s) != cudaSuccess) return MQ_ECUDA;
    if (err_bits) *err_bits = v;
    return v ? MQ_EDEVICE : MQ_OK;
}

}  // namespace

extern "C" int moe_quant_status(const mq_layer_cfg* cfg, int32_t n_tokens, const void* workspace, size_t ws_bytes,
                                uint32_t* err_bits, void* stream) {
    return read_status(cfg, n_tokens, workspace, ws_bytes, err_bits, stream);
}

extern "C" int moe_quant_status_noalloc(const mq_layer_cfg* cfg, int32_t n_tokens, uint32_t* err_bits,
                                        void* stream) {
    const int rc = check_cfg(cfg);
    if (rc != MQ_OK) return rc;
    if (n_tokens < 0 || n_tokens > 65536) return MQ_ESHAPE;
    if (workspace_plan(dims_of(cfg, n_tokens), nullptr, nullptr) > kNoAllocScratchBytes) return MQ_ERANGE;
    void* scratch = nullptr;
    const int sr = noalloc_scratch(&scratch);
    if (sr != MQ_OK) return sr;
    return read_status(cfg, n_tokens, scratch, kNoAllocScratchBytes, err_bits, stream);
}

extern "C" int mq_test_fail_next_decode(uint64_t wait_ns) {
    if (wait_ns == 0 || wait_ns > 1000000000ull) return MQ_EINVAL;
    std::lock_guard<std::mutex> lk(g_wait_test_mu);
    g_wait_test_ns = wait_ns;
    return MQ_OK;
}

extern "C" int mq_unpack_device(int fmt, const void* src, int64_t rows, int64_t cols, float* dst, void* stream) {
    if (!valid_format(fmt)) return MQ_EFORMAT;
    if (rows < 0 || cols < 0) return MQ_EINVAL;
    if (rows * cols == 0) return MQ_OK;
    if (!src || !dst) return MQ_EINVAL;
    if (!aligned16(src)) return MQ_EALIGN;
    if (launch_unpack(fmt, static_cast<const uint8_t*>(src), rows, cols, dst, static_cast<cudaStream_t>(stream)) !=
        cudaSuccess)
        return MQ_ECUDA;
    return MQ_OK;
}

extern "C" int mq_profile_enable(int32_t max_launches) {
    std::lock_guard<std::mutex> lk(g_prof_mu);
    if (max_launches < 0) return MQ_EINVAL;
    for (auto& r : g_prof) { cudaEventDestroy(r.a); cudaEventDestroy(r.b); }
    g_prof.clear();
    g_prof.reserve((size_t)max_launches);
    g_prof_cap = max_launches;
    g_prof_on = max_launches > 0;
    return MQ_OK;
}

extern "C" int mq_profile_collect(mq_kernel_stat* out, int32_t max) {
    std::lock_guard<std::mutex> lk(g_prof_mu);
    std::vector<mq_kernel_stat> agg;
    for (auto& r : g_prof) {
        cudaEventSynchronize(r.b);
        float ms = 0.0f;
        cudaEventElapsedTime(&ms, r.a, r.b);
        size_t i = 0;
        for (; i < agg.size(); ++i)
            if (std::strcmp(agg[i].name, r.name) == 0) break;
        if (i == agg.size()) {
            mq_kernel_stat st;
            std::memset(&st, 0, sizeof(st));
            std::strncpy(st.name, r.name, sizeof(st.name) - 1);
            agg.push_back(st);
        }
        agg[i].launches += 1;
        agg[i].total_ms += ms;
        cudaEventDestroy(r.a);
        cudaEventDestroy(r.b);
    }
    g_prof.clear();
    g_prof_on = false;
    g_prof_cap = 0;
    const int n = (int)agg.size() < max ? (int)agg.size() : max;
    for (int i = 0; i < n && out; ++i) out[i] = agg[i];
    return n;
}
