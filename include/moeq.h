/*
 * moeq — quantized MoE expert-FFN layer for GB300 (sm_103a), C ABI.
 *
 * Computes one DeepSeek-V3-shaped MoE layer whose expert weights are stored
 * in block-quantized, mixed-precision formats, as deployed by the
 * collaborative-compression recipe of arXiv 2509.25689:
 *   - routed experts pruned to a surviving set of E experts (Sec. 3.1),
 *   - sigmoid router scores plus a selection bias, grouped top-k with
 *     topk_group kept groups over the pruned experts and
 *     num_experts_per_tok = k experts per token (Sec. 3.2),
 *   - each expert tensor stored in its own k-quant style format
 *     (Q2_K/Q3_K/Q4_K/Q6_K), Q8_0, or kept unquantized in bf16 (Sec. 3.3,
 *     the planner's level ladder; Sec. 4.1 implementation details),
 *   - SwiGLU expert FFNs, router-weighted combine and an always-on shared
 *     expert (Fig. 1, framework overview of Sec. 3).
 *
 * Conventions (every entry point):
 *   - Plain pointers and sizes.  "device" pointers are CUDA global memory on
 *     the current device; "host" pointers are ordinary CPU memory.
 *   - The caller owns every buffer.  The library keeps no allocation between
 *     calls; scratch comes from the caller's workspace.
 *   - Calls that take a stream enqueue work on it (cudaStream_t passed as
 *     void*, NULL = legacy default stream) and return without waiting.  A
 *     call is not thread-safe with respect to other calls on the same stream.
 *   - Return value: MQ_OK (0) or a negative MQ_E* code; nothing throws.
 *     Argument checks happen on the host before any launch: on error no work
 *     is enqueued.  MQ_ECUDA reports a launch error (cudaGetLastError).
 *
 * Packed tensor format (all formats): a tensor has `rows` output rows and
 * `cols` contraction columns.  Each row is cut into blocks of QK weights
 * along the columns (QK = 256 for Q2_K/Q3_K/Q4_K/Q6_K, 32 for Q8_0 and
 * BF16), the last
 * block padded with zero weights, and rows are padded with zero rows to a
 * multiple of 32 (a tile).  Every field of a block lives in its own plane,
 * starting at a multiple of 256 bytes from the tensor base.  A field's
 * record (the field of one row and one block) is stored in units of at most
 * 64 bytes (the Q4_K and Q6_K 4-bit codes have two units), and unit u of
 * the record of
 * (row r, block b) sits at byte
 *   ((((r / 32) * nb + b) * nu + u) * 32 + r % 32) * unit_bytes
 * of its plane (nb blocks per row, nu units per record), so any block range
 * of a 32-row tile is one contiguous byte range of every plane.  Planes:
 *   Q4_K: d fp16 | dmin fp16 | 12 B sub-scale/min (8 x (6+6) bits) | 128 B 4-bit codes
 *         w = (d*sc)*q - dmin*m,        sub-blocks of 32
 *   Q2_K: d fp16 | dmin fp16 | 16 B (sc | m<<4) per sub-block | 64 B 2-bit codes
 *         w = (d*sc)*q - dmin*m,        sub-blocks of 16
 *   Q3_K: d fp16 | 12 B 6-bit sub-scales (stored sc+32) | 64 B low 2 bits | 32 B high bit
 *         w = (d*(s-32))*(q-4),         sub-blocks of 16
 *   Q8_0: d fp16 | 32 B codes stored as q+128,  w = d*q
 *   Q6_K: d fp16 | 16 B 8-bit sub-scales (stored sc+128) | 128 B low 4 bits
 *         of q | 64 B high 2 bits of q,
 *         w = (d*(s-128))*(q-32),       sub-blocks of 16
 *   BF16: 64 B: the block's 32 weights as bf16, weight k at 16-bit slot
 *         8((k%8)/2) + 2(k/8) + k%2,  w = the bf16 value
 * Inside a block, weight k is in sub-block j = k/n (n = 16 for 2-bit and
 * 1-bit codes and for the Q6_K low 4 bits, 32 for Q4_K and 8-bit codes) at
 * pair m = (k%n)/2, e = k%2.  Codes are little-endian 32-bit words ("pair
 * order"):
 *   2-bit: word 4(j%4) + j/4,          bit 16e + 2m   (Q2_K; Q3_K low bits;
 *                                                      Q6_K high bits)
 *   1-bit: word 2(j%4) + j/8,          bit 16e + 8((j/4)%2) + m
 *   4-bit: word 16(j/4) + 4(j%4) + m/4, bit 16e + 4(m%4)   (Q4_K)
 *   Q6_K 4-bit: word 16(j/8) + 4(j%4) + 2((j/4)%2) + m/4, bit 16e + 4(m%4)
 *   8-bit: word m/2,                   bit 16e + 8(m%2)
 * Sub-block j of Q2_K/Q3_K/Q6_K sits in slot u = 4((j%8)/2) + 2(j/8) + j%2:
 *   Q2_K: byte u = sc | m << 4.
 *   Q6_K: byte u = sc + 128.
 *   Q3_K: bits 4u..4u+3 of bytes 0-7 (LE) = low nibble of s,
 *         bits 2u..2u+1 of bytes 8-11 (LE) = high two bits of s.
 * Q4_K sub-block j (< 8): byte j = (sc & 15) | (m & 15) << 4; bits 4j..4j+1
 *   of bytes 8-11 (LE) = sc >> 4, bits 4j+2..4j+3 = m >> 4.
 * These are this library's own "-style" layouts; the paper defers layouts to
 * llama.cpp and they are not GGUF byte-compatible.  Every decoded weight is
 * exact in fp32 except for the single rounding of the final subtraction
 * (Q2_K/Q4_K) or product (Q6_K: d*(s-128) is exact, its product with q-32
 * is rounded once).
 */
#ifndef MOEQ_H
#define MOEQ_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum { MQ_Q2_K = 1, MQ_Q3_K = 2, MQ_Q4_K = 3, MQ_Q8_0 = 4, MQ_Q6_K = 5, MQ_BF16 = 6 } mq_format;

enum {
    MQ_OK = 0,
    MQ_EINVAL = -1,     /* null pointer, negative size, bad enum */
    MQ_EFORMAT = -2,    /* unknown format code in fmt_per_tensor / fmt */
    MQ_EALIGN = -3,     /* a packed tensor or activation pointer not 16-byte aligned */
    MQ_ESHAPE = -4,     /* inconsistent layer shape (see moe_quant_forward) */
    MQ_EWORKSPACE = -5, /* workspace missing or smaller than moe_quant_workspace_size */
    MQ_ECUDA = -6,      /* CUDA launch or runtime error */
    MQ_EDEVICE = -7,    /* a kernel gave up a bounded wait (see moe_quant_status) */
    MQ_ERANGE = -8,     /* size beyond a documented maximum */
};

/* Layer hyper-parameters.  n_experts = surviving routed experts E after
 * pruning (Sec. 3.1: top ceil(rE) experts kept); top_k = num_experts_per_tok
 * and topk_group = kept groups (Sec. 3.2).  Groups are n_groups contiguous
 * runs of E/n_groups pruned experts.  routed_scale multiplies the
 * normalised routing weights (1.0 = plain normalisation). */
typedef struct {
    int32_t hidden, inter, n_experts, n_groups, topk_group, top_k;
    float routed_scale;
    int32_t has_shared;
} mq_layer_cfg;

/* Device pointers to one expert's packed tensors: gate and up are
 * [inter rows x hidden cols], down is [hidden rows x inter cols]. */
typedef struct { const void* gate; const void* up; const void* down; } mq_expert_weights;

/* experts: HOST array of n_experts entries; shared: HOST pointer to the
 * shared expert's entry, or NULL when cfg.has_shared == 0. */
typedef struct {
    const mq_expert_weights* experts;
    const mq_expert_weights* shared;
} mq_expert_table;

/* Bytes of a packed rows x cols tensor in format fmt (0 on bad arguments). */
size_t mq_packed_size(int fmt, int64_t rows, int64_t cols);

/* Host quantizer (Sec. 3.3 quantizes tensors to a block format; the rule is
 * this library's deterministic nearest-grid rule).  w: host fp32
 * [rows, cols] row-major, finite (for BF16: rounding to a finite bf16);
 * dst: host buffer of dst_bytes >= mq_packed_size.  Returns MQ_OK,
 * MQ_EINVAL (incl. non-finite w) or MQ_EFORMAT. */
int mq_pack(int fmt, const float* w, int64_t rows, int64_t cols, void* dst, size_t dst_bytes);

/* Host dequantizer: src host packed tensor -> dst host fp32 [rows, cols]
 * (padding columns dropped). */
int mq_unpack(int fmt, const void* src, int64_t rows, int64_t cols, float* dst);

/* Device dequantizer: src device packed tensor (16-byte aligned) -> dst
 * device fp32 [rows, cols], stream-ordered.  Bit-identical to mq_unpack. */
int mq_unpack_device(int fmt, const void* src, int64_t rows, int64_t cols, float* dst, void* stream);

/* Workspace bytes moe_quant_forward / moe_quant_route need for n_tokens
 * tokens (0 on invalid cfg).  The workspace must be 256-byte aligned. */
size_t moe_quant_workspace_size(const mq_layer_cfg* cfg, int32_t n_tokens);

/* One MoE layer forward (the hot path).
 *   x              device bf16 [n_tokens, hidden] row-major, 16-byte aligned
 *   router_w       device fp32 [n_experts, hidden] row-major
 *   bias           device fp32 [n_experts] selection bias, or NULL (= 0)
 *   expert_table   host table of device tensor pointers (each 16-byte aligned)
 *   fmt_per_tensor host uint8 [(n_experts + has_shared) * 3]: gate, up, down
 *                  format of every expert, shared expert last
 *   out            device fp32 [n_tokens, hidden]
 *   topk_idx       device int32 [n_tokens, top_k] or NULL: selected pruned
 *                  expert ids, descending biased score, ties to lower id
 *   topk_w         device fp32 [n_tokens, top_k] or NULL: combine weights
 *   workspace      device scratch of ws_bytes >= moe_quant_workspace_size
 * Routing follows a canonical fp32 order so expert ids are bit-exact with
 * the CPU reference; out is fp32 with fp32 accumulation.
 * Range: any finite bf16 token is accepted.  The decode kernels scale every
 * 32-element block of a token (and of the SwiGLU output) by its own power of
 * two; the prefill grouped GEMM (n_tokens >= 64 by default) takes each token
 * as fp16(x * 2^-e), e the exponent of the token's largest |x|, and its
 * SwiGLU output as fp16(h * 2^-2e), undoing both in fp32.  A prefill SwiGLU
 * output still beyond the fp16 range after that scaling (it needs
 * |h| > 65504 * 2^2e, far outside trained models) is not passed on silently:
 * the call's error word gets bit 16 and moe_quant_status returns
 * MQ_EDEVICE.  Weights: the decode kernels take every format's decoded
 * values as they are (BF16 tensors as bf16 MMA operands, the token or h
 * split into bf16 hi + lo); the prefill grouped GEMM decodes weights to
 * fp16, which holds every BF16 weight with 2^-14 <= |w| < 65520 exactly
 * (smaller ones to the nearest fp16 subnormal); a BF16 weight of |w| >=
 * 65520 sets bit 64 of the error word instead.  The tcgen05 decode GEMV
 * (mq_set_path mode 3) takes Q2_K/Q3_K/Q4_K/Q8_0 only: a layer with a
 * Q6_K or BF16 tensor is refused there (MQ_EFORMAT) and, when that kernel
 * would be chosen automatically (hidden or inter not a multiple of 256),
 * runs on the grouped GEMM instead.
 * Shape rules (MQ_ESHAPE): hidden and inter multiples of 128 (hidden <=
 * 32768, inter <= 16384), 1 <= n_experts <= 256, n_experts % n_groups == 0,
 * n_groups <= 64, 1 <= topk_group <= n_groups, 1 <= top_k <= 32 and
 * top_k <= topk_group * n_experts / n_groups, 0 <= n_tokens <= 65536. */
int moe_quant_forward(const mq_layer_cfg* cfg, int32_t n_tokens, const void* x,
                      const float* router_w, const float* bias,
                      const mq_expert_table* expert_table, const uint8_t* fmt_per_tensor,
                      float* out, int32_t* topk_idx, float* topk_w,
                      void* workspace, size_t ws_bytes, void* cuda_stream);

/* moe_quant_forward without a workspace argument, for callers that cannot
 * allocate device memory: plugins and embedding runtimes whose host owns
 * every allocation (they hand out no device buffers of their own), or
 * latency-bound serving loops that must not call cudaMalloc/cudaFree, which
 * can synchronize the whole device.  The paper has no counterpart; it is a
 * deployment convenience of this library.
 *   Arguments, layouts and results are those of moe_quant_forward.
 *   Scratch: a fixed 16 MiB device array inside this library, held on every
 *   device that loads it until the process exits.  A call whose
 *   moe_quant_workspace_size(cfg, n_tokens) exceeds 16 MiB returns MQ_ERANGE
 *   and enqueues nothing (a V3-shaped layer, hidden 7168 / inter 2048 /
 *   top-8 + shared expert, fits up to 29 tokens).
 *   The first call on a device looks the array's device address up
 *   (cudaGetSymbolAddress, with that device current); make that first call
 *   before any stream capture.  It allocates nothing itself.
 *   All calls share the one array and each call overwrites it: calls that
 *   overlap on the GPU (different streams, or several host threads) race
 *   and give wrong results.  Order them on one stream.
 *   Returns the codes of moe_quant_forward, plus MQ_ERANGE as above and
 *   MQ_ECUDA if the address lookup fails. */
int moe_quant_forward_noalloc(const mq_layer_cfg* cfg, int32_t n_tokens, const void* x,
                              const float* router_w, const float* bias,
                              const mq_expert_table* expert_table, const uint8_t* fmt_per_tensor,
                              float* out, int32_t* topk_idx, float* topk_w, void* cuda_stream);

/* Result of the device-side checks of the last moe_quant_forward call made
 * with this workspace and the same cfg / n_tokens.  The expert-FFN kernels
 * give up a wait on a pipeline barrier after a time limit instead of
 * hanging; they then set a bit in an error word of the workspace (cleared at
 * the start of every forward call) and their outputs are not valid.  Bits:
 * 1 / 2 a decode GEMV consumer / producer gave up a wait, 32 a decode down
 * item gave up waiting for its expert's SwiGLU output, 4 a prefill GEMM
 * wait, 8 a tcgen05 GEMV wait, 16 a prefill SwiGLU output beyond the fp16
 * range, 64 a BF16 weight beyond the prefill GEMM's fp16 range (see
 * moe_quant_forward).  This call
 * waits for the stream (cudaStreamSynchronize), reads the word and returns
 * MQ_OK (0 bits), MQ_EDEVICE (some bit set; err_bits, or NULL, receives the
 * bits), or the argument codes of moe_quant_forward (MQ_EWORKSPACE for a
 * workspace that does not fit cfg / n_tokens) and MQ_ECUDA.  n_tokens = 0
 * returns MQ_OK without touching the device.  Not for use while the stream
 * is being captured. */
int moe_quant_status(const mq_layer_cfg* cfg, int32_t n_tokens, const void* workspace, size_t ws_bytes,
                     uint32_t* err_bits, void* cuda_stream);

/* moe_quant_status for moe_quant_forward_noalloc: reads the error word of
 * the library's fixed scratch (same cfg / n_tokens as that call). */
int moe_quant_status_noalloc(const mq_layer_cfg* cfg, int32_t n_tokens, uint32_t* err_bits, void* cuda_stream);

/* Routing and permutation only (steps 1-2 of the layer):
 *   topk_idx/topk_w device [n_tokens, top_k] (required),
 *   offsets  device int32 [n_experts + 1]: exclusive prefix of per-expert counts,
 *   perm     device int32 [n_tokens * top_k]: entry ids (token*top_k + slot)
 *            sorted by (expert, entry id),
 *   inv      device int32 [n_tokens * top_k]: position of each entry in perm.
 * Any of offsets/perm/inv may be NULL. */
int moe_quant_route(const mq_layer_cfg* cfg, int32_t n_tokens, const void* x,
                    const float* router_w, const float* bias,
                    int32_t* topk_idx, float* topk_w, int32_t* offsets, int32_t* perm,
                    int32_t* inv, void* workspace, size_t ws_bytes, void* cuda_stream);

/* Human-readable text of a status code (static string). */
const char* mq_strerror(int status);

/* Path selection: 0 = automatic (n_tokens >= threshold -> prefill grouped
 * GEMM, else decode GEMV), 1 = force decode, 2 = force prefill, 3 = force
 * decode on the alternative tcgen05 GEMV kernels (A operand in tensor
 * memory; slower than the default mma.sync GEMV at decode sizes, kept as a
 * second implementation).  Decode on a layer whose hidden or intermediate
 * size is not a multiple of 256 always takes the tcgen05 GEMV kernels (the
 * mma.sync kernels stream whole 256-element superblocks).  Process wide;
 * the MQ_FORCE_PATH environment variable ("decode"/"prefill"/"decode_tc")
 * sets the initial value.  threshold <= 0 keeps the current one (default
 * 50).  Returns MQ_EINVAL for another mode. */
int mq_set_path(int mode, int32_t prefill_threshold);

/* Test hook for the bounded waits (no counterpart in the paper).  Arms a
 * one-shot fault for the next decode call that runs the default (mma.sync)
 * GEMV kernels: every limit on a pipeline wait becomes wait_ns (0 < wait_ns
 * <= 1e9) and the gate/up kernel's producer posts nothing for its first
 * stage, so the consumers' wait on that stage runs out.  The kernels then
 * record the give-up in the call's error word and exit normally (no copy is
 * left in flight); moe_quant_status reports MQ_EDEVICE, the call's outputs
 * are not valid, and later calls are unaffected.  Process wide; returns
 * MQ_EINVAL for wait_ns out of range. */
int mq_test_fail_next_decode(uint64_t wait_ns);

/* Kernel timing for measurement tools.  mq_profile_enable(n) makes the next
 * calls record a CUDA event pair around each kernel they launch (up to n
 * launches in total; events are created here, host-side).  mq_profile_collect
 * waits for them, writes per-kernel aggregates (up to max entries) and
 * disables recording; returns the number of entries.  Not for use while a
 * stream is being captured. */
typedef struct { char name[48]; int32_t launches; double total_ms; } mq_kernel_stat;
int mq_profile_enable(int32_t max_launches);
int mq_profile_collect(mq_kernel_stat* out, int32_t max);

#ifdef __cplusplus
}
#endif
#endif
