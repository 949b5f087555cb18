// Internal declarations shared by the library's translation units.
#pragma once
#include <cuda_runtime.h>
#include <stdint.h>

#include <cuda_fp16.h>

#include "mq_layout.h"

namespace mq {

// Device pointers and formats of every expert of a layer, passed to kernels
// by value (kernel parameter space) so a forward needs no host->device copy
// and can be captured in a CUDA graph.  Index kMaxExperts... is not used:
// the shared expert sits at index E (n_experts).
struct ExpertTab {
    const uint8_t* p[kMaxExperts + 1][3];
    uint8_t fmt[kMaxExperts + 1][3];
};

struct Dims {
    int H, I, E, G, Gk, K, T;
    int has_shared;
    float routed_scale;
    int x_fams;   // activation families prepared for the tokens (mq_actprep.cuh)
};

// Decode work plan: the expert-FFN kernels cut work into items of 32 rows x
// full K x up to kDecodeTok tokens (gate/up items cover both tensors).  The
// permutation kernel counts items per expert slot (shared expert first, then
// the active routed experts in id order) so the kernels can map an item id to
// its slot.
constexpr int kDecodeTok = 4;
struct Plan {
    int32_t n_slots;
    int32_t dn_target;            // token groups summed over slots
    int32_t ntg_max;              // token groups of the largest slot
    int32_t pad;
    int32_t pre_gu[kMaxExperts + 2];
    int32_t pre_dn[kMaxExperts + 2];
    // per slot: expert id (E = shared), first entry of its tokens in perm, token count
    int32_t slot_e[kMaxExperts + 2];
    int32_t slot_first[kMaxExperts + 2];
    int32_t slot_ntot[kMaxExperts + 2];
};

// Carved out of the caller's workspace (see workspace_plan).
struct Work {
    float* z;          // [T, E] router logits
    int32_t* idx;      // [T, K]
    float* wts;        // [T, K]
    int32_t* offsets;  // [E + 1]
    int32_t* perm;     // [T*K]
    int32_t* inv;      // [T*K]
    int32_t* active;   // [E + 2]: active[0] = count, active[1..] = expert ids
    Plan* plan;        // decode work plan
    __half* xq;        // [T][4][nsb(H)*256] prepared token activations (fp16 fragments)
    float* xs;         // [T][32*nsb(H)] their statistics
    __half* hq;        // [A][4][nsb(I)*256] prepared SwiGLU outputs, A = T*K + T
    float* hs;         // [A][32*nsb(I)]
    float* pdn;        // [A][H] down outputs per assignment (combined by a last pass)
    uint32_t* counters;  // item counters and last-arriver counts (zeroed per call)
    size_t counter_bytes;
    uint32_t* logits_done;  // logits CTAs that published their logits and prepared tokens (zeroed per call)
    uint32_t* route_ready;  // set (release) once the routing result is written (zeroed per call)
    uint32_t* err;     // device error word (bounded waits that ran out)
    __half* x16;       // [T][H] tokens in fp16 for the prefill GEMM (shares xq's bytes),
                       // each token scaled by 2^-xe[t]
    int32_t* xe;       // [T] per-token power-of-two exponents of x16 (prefill path)
    __half* h16;       // [A][I] fp16 SwiGLU outputs for the prefill GEMM (shares hq's bytes)
    float* spart;         // decode: the shared expert's gate/up K halves [T][2][2][I]
    uint32_t* zero_words; // counters + error word, cleared by the first kernel of a call
    int n_zero;
};

size_t workspace_plan(const Dims& d, void* base, Work* w);

// Per-device one-time set-up.  Function attributes (shared-memory limits,
// carveout preference) apply to one device, so a translation unit's set-up
// runs once for every device it is used on: device_setup(slot, init) runs
// init() the first time `slot` is used with the current device (under a
// process-wide mutex) and returns that device's SM count (0 if the device
// query failed).  Slots: one per translation unit or kernel group.
enum SetupSlot : int { kSetupDecode = 0, kSetupPrefill, kSetupTgemv, kSetupRoute, kSetupCombine, kSetupStats,
                 kSetupSlots };
int device_setup(int slot, void (*init)());

// Test hook of the bounded waits (mq_test_fail_next_decode): true once after
// it was armed, with the shortened wait limit in *wait_ns.
bool take_wait_test(uint64_t* wait_ns);

// launch helpers; each returns cudaGetLastError() of its launch
// Programmatic dependent launch: every kernel of the layer is launched with
// programmatic stream serialization, waits for its predecessor's results
// with pdl_wait() before touching global memory, and lets its successor be
// scheduled early with pdl_launch().
#ifdef __CUDACC__
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_launch() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }

template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t s,
                       Args... args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kernel, static_cast<KArgs>(args)...);
}

// The small kernels of a layer call ask for the largest shared-memory
// carveout as the FFN kernels (227 KB per CTA) need it, so an SM keeps one
// L1/shared split across the call instead of switching between kernels.
template <typename... KArgs>
void prefer_max_shared(void (*kernel)(KArgs...)) {
    cudaFuncSetAttribute(kernel, cudaFuncAttributePreferredSharedMemoryCarveout, (int)cudaSharedmemCarveoutMaxShared);
}
#endif

// Routing fused into the logits kernel (decode path): the CTA that finishes
// last routes every token and permutes (idx/wts/offsets/perm/inv/active/plan
// as the permutation kernel writes them), then sets route_ready with a
// release store; every CTA first counts itself in logits_done after its
// logits and prepared tokens are written.  Both words must be zero at launch.
struct FusedRoute {
    int on;
    uint32_t n_ctas;          // filled in by the launcher
    Dims d;
    const float* bias;
    int32_t* idx; float* wts; int32_t* offsets; int32_t* perm; int32_t* inv; int32_t* active;
    Plan* plan;
    uint32_t* logits_done;
    uint32_t* route_ready;
};

// Clears n words (the per-call counters) once the previous kernel on the
// stream is done; the first kernel of every forward call.
cudaError_t launch_zero(uint32_t* words, int n, cudaStream_t s);
// fused: nullptr, or the routing outputs for the fused last-CTA routing
// (the logits kernel with activation prep; router_logits_ctas(d) CTAs, each
// up to 4 experts x 8 tokens)
cudaError_t launch_router_logits(const Dims& d, const uint16_t* x, const float* W, float* z, __half* xq, float* xs,
                                 __half* x16, int32_t* xe, const FusedRoute* fused, cudaStream_t s);
uint32_t router_logits_ctas(const Dims& d);
cudaError_t launch_topk(const Dims& d, const float* z, const float* bias, int32_t* idx, float* wts, cudaStream_t s);
cudaError_t launch_permute(const Dims& d, const int32_t* idx, int32_t* offsets, int32_t* perm, int32_t* inv,
                           int32_t* active, Plan* plan, cudaStream_t s);
cudaError_t launch_route_permute(const Dims& d, const float* z, const float* bias, int32_t* idx, float* wts,
                                 int32_t* offsets, int32_t* perm, int32_t* inv, int32_t* active, Plan* plan,
                                 cudaStream_t s);
cudaError_t launch_combine(const Dims& d, const float* pdn, float* out, cudaStream_t s);
cudaError_t launch_prefill(const Dims& d, const ExpertTab& tab, const Work& w, float* out, cudaStream_t s);
cudaError_t launch_decode_mma(const Dims& d, const ExpertTab& tab, const Work& w, float* out, cudaStream_t s);
// tcgen05 decode kernels: need hidden and inter to be multiples of 128
bool decode_tc_fits(const Dims& d);
// mma.sync decode kernels: stream whole 256-element superblocks of every
// format (a Q8_0 stage holds 8 blocks of 32 per superblock), so hidden and
// inter must be multiples of 256; other shapes take the tcgen05 decode kernels
bool decode_mma_fits(const Dims& d);
cudaError_t launch_decode_tc(const Dims& d, const ExpertTab& tab, const Work& w, float* out, cudaStream_t s);
size_t decode_counter_bytes(const Dims& d);
cudaError_t launch_unpack(int fmt, const uint8_t* src, int64_t rows, int64_t cols, float* dst, cudaStream_t s);

// kernel timing hooks (no-ops unless profiling is enabled)
void prof_begin(const char* name, cudaStream_t s);
void prof_end(cudaStream_t s);

}  // namespace mq
