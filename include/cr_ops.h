/*
 * cr_ops.h - the kernels inside the four cr.h calls, exposed one by one so
 * that each step of the repair path can be checked on its own.  Same
 * conventions as cr.h (caller-owned device buffers, 16-byte alignment,
 * asynchronous on `stream`, host-side validation, no allocation).
 */
#ifndef CR_OPS_H_
#define CR_OPS_H_

#include "cr.h"

#ifdef __cplusplus
extern "C" {
#endif

/* Epilogues of cr_linear. */
typedef enum cr_linear_epi {
    CR_EPI_BF16 = 0,      /* out(bf16)  = A W^T + bias                         */
    CR_EPI_GELU_BF16 = 1, /* out(bf16)  = GELU_erf(A W^T + bias)  (MLP, R4)    */
    CR_EPI_ADD_F32 = 2,   /* out(fp32) += A W^T + bias      (residual stream)  */
    CR_EPI_F32 = 3        /* out(fp32)  = A W^T + bias                         */
} cr_linear_epi;

/*
 * cr_linear - out = epi(A W^T + bias) on the tcgen05 tensor cores, bf16
 * operands, fp32 accumulation (every linear of Sec. 4.1).
 * A [M, K] bf16 with row stride lda elements; W [N, K] bf16 (row stride K);
 * bias [N] fp32 or NULL; out [M, N] with row stride ldo elements.
 * K must be a multiple of 8; M, N >= 1.
 */
cr_status cr_linear(const uint16_t* A, int64_t lda, const uint16_t* W, const float* bias,
                    int64_t M, int64_t N, int64_t K, void* out, int64_t ldo, int32_t epi,
                    void* stream);

/*
 * cr_matmul - the matrix products of the training step's backward pass
 * (Sec. 4.2; App. A optimisation): dX = dY W and dW = dY^T X, on the tcgen05
 * tensor cores with bf16 operands and fp32 accumulation:
 *   C = op(A) B,  or  C += op(A) B  if accumulate != 0.
 * B [K, N] bf16, row stride ldb (N contiguous).  op(A) [M, K]: A stored
 * [M, K] (a_trans = 0) or A stored [K, M] and transposed (a_trans = 1), row
 * stride lda.  C [M, N] fp32, row stride ldc.  N must be a multiple of 64, and
 * so must M when a_trans; lda and ldb multiples of 8, ldc of 4; pointers
 * 16-byte aligned.  workspace: NULL, or fp32 scratch of workspace_bytes (16-byte
 * aligned) that lets a product whose tiles fill the GPU poorly run as up to 8
 * k-parts (each written to the scratch, then summed in a fixed order into C:
 * deterministic, a different rounding order than one k-loop).  Errors:
 * CR_ERR_INVALID_ARG for non-positive sizes, bad strides or pointers;
 * CR_ERR_UNSUPPORTED for widths that are not whole 64-column blocks.
 */
cr_status cr_matmul(const uint16_t* A, int64_t lda, int32_t a_trans, const uint16_t* B, int64_t ldb,
                    int64_t M, int64_t N, int64_t K, float* C, int64_t ldc, int32_t accumulate,
                    void* workspace, size_t workspace_bytes, void* stream);

/*
 * cr_layernorm - u = LN(x + add) * gamma + beta per row (biased variance,
 * eps), fp32 statistics (R4).  x [M, D] fp32 (row stride D).  If `add` is
 * non-NULL ([M, D] fp32, row stride ld_add, a multiple of 4), x + add is also
 * written to x_out ([M, D] fp32; may equal x).  u [M, D] bf16.  D a multiple
 * of 128, at most 1024.
 */
cr_status cr_layernorm(const float* x, const float* add, int64_t ld_add, float* x_out,
                       const float* gamma, const float* beta, float eps, int64_t M, int64_t D,
                       uint16_t* u, void* stream);

/*
 * cr_chunk_causal_attention - softmax(Q K^T / sqrt(d) masked to
 * c(j) <= c(i)) V per head and request (Sec. 4.1, block-causal mask).
 * qkv [N, 3 d_b] bf16: Q at columns [0, d_b), K at [d_b, 2 d_b), V at
 * [2 d_b, 3 d_b); head h at h*d .. (h+1)*d inside each (d = d_b / n_heads,
 * 32 or 64; RoPE already applied).  chunk_end [N] int32 (request-local
 * exclusive end of each token's chunk; key j is visible to query i iff
 * j < chunk_end[i]).  cu_seqlens_host [n_req + 1] HOST.  out [N, d_b] bf16.
 */
cr_status cr_chunk_causal_attention(const uint16_t* qkv, int32_t d_b, int32_t n_heads,
                                    const int32_t* chunk_end, const int32_t* cu_seqlens_host,
                                    int32_t n_req, int64_t n_tokens, uint16_t* out,
                                    void* stream);

/*
 * cr_masked_attention - the same attention under any cr_mask_mode (Sec. 4.1
 * for A0, App. F for the ablations A1-A3).  Arguments as in
 * cr_chunk_causal_attention, plus: chunk_end is read for
 * CR_MASK_BLOCK_CAUSAL and CR_MASK_BLOCK_DIAGONAL (may be NULL otherwise);
 * chunk_start [N] int32 (request-local start of each token's chunk, as
 * written by cr_chunk_starts) is read for CR_MASK_BLOCK_DIAGONAL only (may be
 * NULL otherwise).  Every query sees at least itself in every mode.
 */
cr_status cr_masked_attention(const uint16_t* qkv, int32_t d_b, int32_t n_heads,
                              int32_t mask_mode, const int32_t* chunk_end,
                              const int32_t* chunk_start, const int32_t* cu_seqlens_host,
                              int32_t n_req, int64_t n_tokens, uint16_t* out, void* stream);

/*
 * cr_chunk_starts - chunk_start[t] = request-local index of the first token
 * of t's chunk, from the chunk map of cr_assemble_stale: the smallest u with
 * chunk_end[u] > t inside t's request (chunk_end is non-decreasing there).
 * chunk_end, chunk_start [N] int32 device; cu_seqlens_host [n_req+1] HOST.
 * Integer work, exact.
 */
cr_status cr_chunk_starts(const int32_t* chunk_end, const int32_t* cu_seqlens_host, int32_t n_req,
                          int64_t n_tokens, int32_t* chunk_start, void* stream);

/*
 * cr_wait_selftest - failure-reporting check: one CTA waits on a pipeline
 * barrier that nothing arrives on, through the bounded wait every kernel of
 * the library uses.  The wait gives up after its limit (2 s), records a
 * timeout at site 900 in the device status word and returns, so
 * cr_get_device_status then returns CR_ERR_TIMEOUT with out = {1, 900, 0}; the
 * context stays usable (cr_clear_device_status resets the word).
 */
cr_status cr_wait_selftest(void* stream);

/*
 * cr_qkv_rope - the repair block's QKV linear with the repairer RoPE fused
 * into its epilogue: qkv = u W_qkv^T + b_qkv, then Q and K of every head
 * rotated (rotate-half pairs, angle pos[t] * theta^(-2i/d)).
 * u [N, d_b] bf16; w_qkv [3 d_b, d_b]; qkv [N, 3 d_b] bf16.
 */
cr_status cr_qkv_rope(const uint16_t* u, const uint16_t* w_qkv, const float* b_qkv,
                      const int32_t* pos, int64_t n_tokens, int32_t d_b, int32_t n_heads,
                      float rope_theta, uint16_t* qkv, void* stream);

/*
 * cr_segment_project - StaleEncoder stage 1 (Sec. 4.1):
 *   y[t, s*d_seg + k] = sum_d W_seg[s,k,d] kv[t, s*d_h + d] / sigma_stale[s*d_h + d]
 *                       + b_seg[s,k]
 * kv [N, D_KV] bf16; y [N, S*d_seg] bf16 (fp32 sums rounded once).  workspace:
 * at least S*d_seg*d_h*4 bytes (holds W_seg with 1/sigma folded in, as two
 * bf16 terms per weight).
 */
cr_status cr_segment_project(const cr_target_dims* target, int32_t d_seg, const uint16_t* kv,
                             int64_t n_tokens, const uint16_t* w_seg, const float* b_seg,
                             const float* sigma_stale, uint16_t* y, void* workspace,
                             size_t workspace_bytes, void* stream);

/*
 * cr_segment_project_noalloc - cr_segment_project without a workspace, for
 * callers that cannot allocate device memory (an engine plugin living inside
 * a fixed, pre-planned memory budget; a serving loop that must never call
 * cudaMalloc, which can synchronise the device).  The paper has no
 * counterpart: this is a deployment variant of the same computation.
 *
 * Its scratch (W_seg with 1/sigma_stale folded in, two bf16 terms for each of
 * the S*d_seg*d_h weights) is a fixed 8 MiB device array inside the library,
 * present on every GPU that loads the library until the process exits: at
 * most S*d_seg*d_h = 2 Mi weights (the 8B-shape target has 1 Mi).  Larger
 * shapes return CR_ERR_UNSUPPORTED.  The first call on a device looks up that array's
 * device address (cudaGetSymbolAddress); make that first call before any
 * stream capture.  All calls share the one array, so calls whose kernels
 * overlap on the GPU (different streams, no ordering between them) race on
 * it; calls on one stream are safe.  Nothing in the array needs clearing:
 * each call rewrites every element it reads.  Nothing is allocated or freed.
 * Arguments, layouts and errors otherwise as cr_segment_project.
 */
cr_status cr_segment_project_noalloc(const cr_target_dims* target, int32_t d_seg,
                                     const uint16_t* kv, int64_t n_tokens, const uint16_t* w_seg,
                                     const float* b_seg, const float* sigma_stale, uint16_t* y,
                                     void* stream);

#ifdef __cplusplus
}
#endif
#endif /* CR_OPS_H_ */
