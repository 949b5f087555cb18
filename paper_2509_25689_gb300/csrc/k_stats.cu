// Device histogram of routed experts and the expert-importance scores of
// performance-aware pruning (arXiv 2509.25689 Sec. 3.1):
//   f_e = count_e / n_tokens, s_e = (sum of e's routing weights) / count_e,
//   I_e = alpha f_e + (1 - alpha) s_e, keep the ceil(r E) largest I_e.
// Every CTA builds a private histogram in shared memory (integer counts and
// 128-bit fixed-point weight sums, mq_fixsum.h) over a grid-stride slice of
// the routed entries, then adds it to the global buffer with integer
// atomics; integer addition makes the result independent of the order.
#include <cuda_runtime.h>

#include <cmath>
#include <cstdint>

#include "../../include/moeq.h"
#include "../../include/moeq_stats.h"
#include "mq_fixsum.h"
#include "mq_internal.h"

namespace mq {
namespace {

constexpr int kMaxStatExperts = 1024;
constexpr int kAddThreads = 512;

struct StatsView {
    unsigned long long* n_tokens;
    unsigned int* err;
    unsigned long long* count;
    unsigned long long* lo;
    unsigned long long* hi;
};

__host__ __device__ inline StatsView stats_view(void* base, int E) {
    uint8_t* b = static_cast<uint8_t*>(base);
    StatsView v;
    v.n_tokens = reinterpret_cast<unsigned long long*>(b);
    v.err = reinterpret_cast<unsigned int*>(b + 8);
    v.count = reinterpret_cast<unsigned long long*>(b + 16);
    v.lo = v.count + E;
    v.hi = v.lo + E;
    return v;
}

// (hi:lo) += (vhi:vlo) with two atomics; the carry out of the low word is
// taken from the value the low-word atomic returned, so the final 128-bit
// value is exact whatever the interleaving.
__device__ __forceinline__ void atomic_add128(unsigned long long* lo, unsigned long long* hi, unsigned long long vlo,
                                              unsigned long long vhi) {
    const unsigned long long old = atomicAdd(lo, vlo);
    atomicAdd(hi, vhi + (old + vlo < old ? 1ull : 0ull));
}

__global__ void __launch_bounds__(kAddThreads) stats_add_kernel(void* stats, int E, const int32_t* __restrict__ idx,
                                                                const float* __restrict__ w, long long n,
                                                                int n_tokens) {
    __shared__ unsigned long long s_cnt[kMaxStatExperts], s_lo[kMaxStatExperts], s_hi[kMaxStatExperts];
    const StatsView g = stats_view(stats, E);
    for (int e = threadIdx.x; e < E; e += blockDim.x) s_cnt[e] = s_lo[e] = s_hi[e] = 0ull;
    __syncthreads();
    unsigned int bad = 0;
    const long long stride = (long long)gridDim.x * blockDim.x;
    for (long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += stride) {
        const int e = __ldg(idx + i);
        const float wv = __ldg(w + i);
        Fix128 f;
        if (e < 0 || e >= E) {
            bad |= 1u;
            continue;
        }
        if (!fix_from_float(wv, f)) {
            bad |= 2u;
            continue;
        }
        atomicAdd(&s_cnt[e], 1ull);
        atomic_add128(&s_lo[e], &s_hi[e], f.lo, f.hi);
    }
    bad = __reduce_or_sync(0xFFFFFFFFu, bad);
    if (bad != 0 && (threadIdx.x & 31) == 0) atomicOr(g.err, bad);
    __syncthreads();
    for (int e = threadIdx.x; e < E; e += blockDim.x) {
        if (s_cnt[e] == 0) continue;
        atomicAdd(g.count + e, s_cnt[e]);
        atomic_add128(g.lo + e, g.hi + e, s_lo[e], s_hi[e]);
    }
    if (blockIdx.x == 0 && threadIdx.x == 0) atomicAdd(g.n_tokens, (unsigned long long)n_tokens);
}

__global__ void __launch_bounds__(kMaxStatExperts) stats_scores_kernel(const void* stats, int E, double alpha, int k,
                                                                       double* freq, double* mean_w, double* scores,
                                                                       int32_t* keep) {
    __shared__ double s_sc[kMaxStatExperts];
    __shared__ int s_warp[kMaxStatExperts / 32];
    const StatsView g = stats_view(const_cast<void*>(stats), E);
    const int e = threadIdx.x, lane = e & 31, warp = e >> 5;
    const unsigned long long nt = *g.n_tokens;
    double I = 0.0;
    if (e < E) {
        const unsigned long long c = g.count[e];
        const double f = nt > 0 ? __ddiv_rn((double)c, (double)nt) : 0.0;
        const double s = c > 0 ? __ddiv_rn(fix_to_double(Fix128{g.lo[e], g.hi[e]}), (double)c) : 0.0;
        I = __dadd_rn(__dmul_rn(alpha, f), __dmul_rn(__dsub_rn(1.0, alpha), s));
        if (freq) freq[e] = f;
        if (mean_w) mean_w[e] = s;
        if (scores) scores[e] = I;
        s_sc[e] = I;
    }
    __syncthreads();
    if (keep == nullptr) return;
    // rank of e: experts with a larger score, or an equal score and a lower id
    int rank = 0;
    if (e < E)
        for (int j = 0; j < E; ++j) {
            const double o = s_sc[j];
            rank += (o > I || (o == I && j < e)) ? 1 : 0;
        }
    const bool kept = e < E && rank < k;
    // kept ids in ascending order: exclusive prefix count of the kept flags
    const unsigned int ball = __ballot_sync(0xFFFFFFFFu, kept);
    if (lane == 0) s_warp[warp] = __popc(ball);
    __syncthreads();
    int pos = __popc(ball & ((1u << lane) - 1u));
    for (int q = 0; q < warp; ++q) pos += s_warp[q];
    if (kept) keep[pos] = e;
}

bool aligned(const void* p, uintptr_t a) { return (reinterpret_cast<uintptr_t>(p) & (a - 1)) == 0; }

void stats_setup() {}

}  // namespace
}  // namespace mq

using namespace mq;

extern "C" size_t mq_expert_stats_bytes(int32_t n_experts) {
    if (n_experts < 1 || n_experts > kMaxStatExperts) return 0;
    return 16 + 24 * (size_t)n_experts;
}

extern "C" int mq_expert_stats_reset(void* stats, int32_t n_experts, void* stream) {
    const size_t bytes = mq_expert_stats_bytes(n_experts);
    if (bytes == 0 || stats == nullptr) return MQ_EINVAL;
    if (!aligned(stats, 16)) return MQ_EALIGN;
    return cudaMemsetAsync(stats, 0, bytes, static_cast<cudaStream_t>(stream)) == cudaSuccess ? MQ_OK : MQ_ECUDA;
}

extern "C" int mq_expert_stats_add(void* stats, int32_t n_experts, const int32_t* topk_idx, const float* topk_w,
                                   int32_t n_tokens, int32_t top_k, void* stream) {
    if (mq_expert_stats_bytes(n_experts) == 0 || stats == nullptr || n_tokens < 0 || top_k < 1 || top_k > 32)
        return MQ_EINVAL;
    if (n_tokens == 0) return MQ_OK;
    if (topk_idx == nullptr || topk_w == nullptr) return MQ_EINVAL;
    if (!aligned(stats, 16) || !aligned(topk_idx, 4) || !aligned(topk_w, 4)) return MQ_EALIGN;
    const int sms = device_setup(kSetupStats, stats_setup);
    if (sms <= 0) return MQ_ECUDA;
    const long long n = (long long)n_tokens * top_k;
    // about 16 entries per thread, at most two CTAs per SM
    const long long want = (n + kAddThreads * 16LL - 1) / (kAddThreads * 16LL);
    const int grid = (int)(want < 2LL * sms ? want : 2LL * sms);
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    prof_begin("expert_stats_add", s);
    stats_add_kernel<<<grid, kAddThreads, 0, s>>>(stats, n_experts, topk_idx, topk_w, n, n_tokens);
    prof_end(s);
    return cudaGetLastError() == cudaSuccess ? MQ_OK : MQ_ECUDA;
}

extern "C" int mq_expert_stats_scores(const void* stats, int32_t n_experts, double alpha, double retain, double* freq,
                                      double* mean_w, double* scores, int32_t* keep, int32_t* n_keep, void* stream) {
    if (mq_expert_stats_bytes(n_experts) == 0 || stats == nullptr) return MQ_EINVAL;
    if (!(alpha >= 0.0 && alpha <= 1.0) || !(retain > 0.0 && retain <= 1.0)) return MQ_EINVAL;
    if (!aligned(stats, 16) || !aligned(freq, 8) || !aligned(mean_w, 8) || !aligned(scores, 8) || !aligned(keep, 4))
        return MQ_EALIGN;
    const int k = (int)std::ceil(retain * n_experts - 1e-12);
    if (n_keep) *n_keep = k;
    if (!freq && !mean_w && !scores && !keep) return MQ_OK;
    if (device_setup(kSetupStats, stats_setup) <= 0) return MQ_ECUDA;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    prof_begin("expert_stats_scores", s);
    stats_scores_kernel<<<1, kMaxStatExperts, 0, s>>>(stats, n_experts, alpha, k, freq, mean_w, scores, keep);
    prof_end(s);
    return cudaGetLastError() == cudaSuccess ? MQ_OK : MQ_ECUDA;
}
