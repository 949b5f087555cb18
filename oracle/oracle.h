/*
 * Oracle for the quantized MoE expert FFN — TEST INFRASTRUCTURE ONLY.
 *
 * A plain, slow, single-threaded CPU restatement of what the GPU path
 * computes: block-format unpack (and the quantizer that defines pack),
 * the canonical fp32 router (sigmoid scores, selection bias, group-limited
 * top-k, normalised weights), the token->expert permutation, and the SwiGLU
 * expert FFN with weighted combine and shared expert in fp64.
 *
 * Only the test suite, the smoke check and the benchmark's CPU-baseline leg
 * may load this library.  It shares no source with the CUDA library: its
 * own layout code, its own fp16 conversion, its own sigmoid.
 *
 * Paper anchors (arXiv 2509.25689):
 *   - MoE block with shared + routed experts and a router: Fig. 1 and the
 *     "Framework Overview" of Sec. 3.
 *   - num_experts_per_tok (k) and topk_group over the pruned expert set:
 *     Sec. 3.2 (Hardware-Aware Activation Adjustment).
 *   - k-quant style block formats (Q2_K/Q3_K/Q4_K/Q6_K) and Q8, and bf16
 *     tensors kept unquantized: Sec. 3.3 (the level ladder of the
 *     precision planner) and the implementation details of Sec. 4.1.  The paper defers the byte
 *     layout to llama.cpp; the layouts here are this project's own
 *     definitions of "-style" formats (not GGUF byte-compatible).
 *
 * Parity status per function is listed in the header comment of oracle.c.
 */
#ifndef MOE_ORACLE_H
#define MOE_ORACLE_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

enum { ORC_Q2_K = 1, ORC_Q3_K = 2, ORC_Q4_K = 3, ORC_Q8_0 = 4, ORC_Q6_K = 5, ORC_BF16 = 6 };

typedef struct {
    int32_t hidden, inter, n_experts, n_groups, topk_group, top_k;
    float routed_scale;
    int32_t has_shared;
} oracle_layer;

/* Bytes of a rows x cols tensor in format fmt (planes 256-byte aligned). */
size_t oracle_packed_size(int fmt, int64_t rows, int64_t cols);

/* Quantize fp32 weights [rows, cols] into dst.  Returns 0 or -1. */
int oracle_pack(int fmt, const float* w, int64_t rows, int64_t cols,
                uint8_t* dst, size_t dst_bytes);

/* Dequantize into dst [rows, cols] fp32 (padding columns dropped). */
int oracle_unpack(int fmt, const uint8_t* src, int64_t rows, int64_t cols,
                  float* dst);

/* Canonical fp32 sigmoid (range reduction + degree-7 Taylor). */
float oracle_sigmoid(float z);

/* Canonical router logit for one (token, expert): x bf16 bits, w fp32. */
float oracle_router_logit(const uint16_t* x, const float* w, int32_t hidden);

/* Route T tokens.  idx/w: [T, k].  z_out/s_out (optional): [T, E]. */
int oracle_route(const oracle_layer* L, int32_t T, const uint16_t* x,
                 const float* router_w, const float* bias, int32_t* idx,
                 float* w, float* z_out, float* s_out);

/* The selection step of oracle_route alone, on precomputed scores: s [T, E]
   (sigmoid scores, e.g. s_out of oracle_route) plus the selection bias ->
   idx/w [T, k].  Lets a caller re-select under other biases without
   recomputing the logits (the logits do not depend on the bias). */
int oracle_select(const oracle_layer* L, int32_t T, const float* s, const float* bias,
                  int32_t* idx, float* w);

/* Stable counting sort of (token, slot) entries by expert.
   offsets [E+1], perm [T*k] (entry ids), inv [T*k] (position of entry). */
int oracle_permute(int32_t T, int32_t k, int32_t E, const int32_t* idx,
                   int32_t* offsets, int32_t* perm, int32_t* inv);

/* Full layer: y [T, H] fp32 (computed in fp64).  gate/up/down: host arrays
   of E(+1 shared) packed-tensor pointers; fmt: [(E+has_shared)*3] formats
   in the order gate, up, down.  idx/w (optional): routing result. */
int oracle_moe_forward(const oracle_layer* L, int32_t T, const uint16_t* x,
                       const float* router_w, const float* bias,
                       const void* const* gate, const void* const* up,
                       const void* const* down, const uint8_t* fmt,
                       float* y, int32_t* idx, float* w);

#ifdef __cplusplus
}
#endif
#endif
