// Internal declarations shared by the library's translation units.
#pragma once
#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "cr.h"
#include "cr_ops.h"

// Device status codes (status word element 0).
enum : unsigned { CR_DEV_OK = 0u, CR_DEV_TIMEOUT = 1u, CR_DEV_INDEX = 2u };

namespace cr {

constexpr int kMaxSegs = 512;   // selected chunks per cr_assemble_stale call
constexpr int kMaxReq = 256;    // requests per call

// ------------------------------------------------------------------ gather
struct GatherSeg {
    int64_t src_row;     // first pool row of the chunk
    int64_t dst_row;     // first output row
    int32_t len;         // rows
    int32_t chunk_local; // c(t) of the chunk inside its request
    int32_t local_start; // request-local position of the chunk's first token
    int32_t pad;
};
struct GatherParams {
    const uint8_t* kv_pool;
    const uint8_t* emb_pool;
    uint8_t* kv_out;
    uint8_t* emb_out;
    int64_t kv_row_bytes;
    int64_t emb_row_bytes;
    int32_t* chunk_id;
    int32_t* chunk_end;
    int32_t* pos;
    int32_t* cu_seqlens;
    int64_t n_tokens;
    int64_t n_pool_tokens;
    unsigned* status;
    int32_t n_seg;
    int32_t n_req;
    int32_t cu_seqlens_host[kMaxReq + 1];
    GatherSeg seg[kMaxSegs];
};

// ------------------------------------------------------------------ GEMM
enum GemmEpi : int {
    EPI_BF16 = 0,
    EPI_GELU_BF16 = 1,
    EPI_ADD_F32 = 2,
    EPI_F32 = 3,
    EPI_QKV_ROPE = 4,   // bf16 out, repairer RoPE on columns < rope_cols
    EPI_KV_BF16 = 5,    // in-place residual add on a bf16 cache tile (+ global RoPE on K)
    EPI_KV_F32 = 6,     // same for an fp32 cache
    EPI_KV_PAGED = 7,   // bf16 cache: stale tile read token-major, repaired rows written
                        // to a paged, layer-major target cache through a slot mapping
    EPI_KV_LOSS = 8,    // training head: r = z + b - (joint - stale) / sigma from the staged
                        // bf16 stale and joint tiles; writes dz = row_scale[t] r (bf16)
                        // and per-row partial sums of r^2 instead of storing r
    EPI_KV_POOL = 9     // EPI_KV_BF16 with the stale tile read from the chunk pool (rows
                        // src_row[t]) and the repaired rows stored into the output cache
};

// Operand layouts of the GEMM: K-major A and W (the forward), K-major A with
// MN-major W (dX = dY W), MN-major A and W (dW = dY^T X).
// LAY_KK2: both operands K-major, two products in one launch (launch_gemm_pair);
// its own instantiation, so that the one-product kernels carry none of its logic
enum GemmLayout : int { LAY_KK = 0, LAY_KM = 1, LAY_MM = 2, LAY_KK2 = 3 };

struct GemmParams {
    int32_t M, N, K;
    int32_t num_m, num_n;
    const float* bias;       // [N] or null
    void* out;               // non-KV epilogues
    int64_t ldo;             // elements
    const int32_t* pos;      // [M] (RoPE epilogues)
    int32_t rope_dim;        // head dim the RoPE pairs live in
    int32_t rope_cols;       // QKV: columns [0, rope_cols) are rotated (Q and K)
    int32_t rope_on;         // KV: rotate K segments
    int32_t n_kv_heads;      // KV: segment s is K iff (s / n_kv_heads) is even
    const float* sigma;      // KV: sigma_delta [N]
    const float2* rope_table;  // QKV: (cos, sin) [rope_dim / 2, M] angle-major, or null (computed inline)
    const int64_t* slot;     // KV_PAGED: destination slot of each token, < 0 = not written
    uint16_t* paged;         // KV_PAGED: [N / seg_width][num_slots][seg_width] bf16
    int64_t num_slots;       // KV_PAGED: slots per (layer, K|V) plane
    int32_t seg_width;       // KV_PAGED: H_kv * d_h, the columns of one (layer, K|V) plane
    // KV output choices (App. F): only the column blocks [b w, (b + 1) w), w =
    // col_block, with b % 2 == col_phase (0: K, 1: V) are visited, or every
    // column if col_block == 0; kv_zero: zero output offset (A5), sigma (z + b)
    // replaces kv + sigma (z + b); rows t with keep_chunk[t] == 0 (the first
    // chunk) keep their stale value, if keep_chunk is given.
    int32_t col_block;
    int32_t col_phase;
    int32_t kv_zero;
    const int32_t* keep_chunk;
    // EPI_KV_LOSS: the stale cache is the in-place tile, the joint cache [M, N] bf16
    // (same row stride) comes in through tm_joint, sigma holds sigma_Delta; dz [M, N]
    // bf16; row_scale [M]; loss_part [2 num_n][M], the sum of r^2 over each
    // (column tile, epilogue column group) of a row
    const uint16_t* loss_joint;
    uint16_t* loss_dz;
    const float* row_scale;
    float* loss_part;
    unsigned* status;
    // two-term A (set by launch_gemm when A_lo is given): A = A_hi + A_lo, both
    // bf16 [M, K]; the k-loop runs over the split_kb k-blocks of A_hi, then the
    // same k-blocks of A_lo (tm_alo) against the same W columns, into one
    // accumulator: A at about 16 significant bits for twice the MMAs.  0 = plain A.
    int32_t split_kb;
    // split-K (launch_gemm_lay): parts per tile, each writing rows [u M, (u + 1) M)
    // of the output (1 = off; every launcher sets it)
    int32_t split_k;
    // tile order: 0 = W-tile-major (row tiles fastest), 1 = column tiles fastest
    // (k-parts slowest), for an A operand far larger than L2
    int32_t n_fast;
    // grouped rows (launch_gemm_lay): every bgroup_rows rows of A form a group whose
    // tile reads W columns [g BN, (g + 1) BN) of the W matrix, g = row / bgroup_rows,
    // and writes output columns [0, BN); 0 = off
    int32_t bgroup_rows;
    // two products in one launch (launch_gemm_pair, EPI_F32): the output columns
    // [n_split, N) of the launch belong to a second product with its own A
    // (tm_a2, two-term through tm_alo2 when split_kb2 > 0), W (tm_b2, its rows
    // counted from n_split), K2, bias2 and output (tm_c2, its columns counted from
    // n_split); n_split is a multiple of the tile width.  0 = one product.
    int32_t n_split;
    int32_t K2;
    int32_t split_kb2;
    const float* bias2;
    // EPI_KV_POOL: the stale cache rows come from the pool (bf16 [n_pool, N], row
    // stride N): box_src[b] the pool row of the first of request rows 128 b ..
    // 128 b + 127 when they are one contiguous pool range (one TMA box through
    // tm_pool), else -1; then grp_src[g] the same for rows 8 g .. 8 g + 7 (one
    // 8-row TMA box through tm_pool8), else -1 (each row from src_row[t])
    const uint16_t* kv_pool;
    const int64_t* src_row;
    const int64_t* box_src;
    const int64_t* grp_src;
    float inv_freq[64];      // RoPE frequencies, rope_dim / 2 entries
    CUtensorMap tm_joint;    // EPI_KV_LOSS (set by launch_gemm; the type carries its alignment)
    CUtensorMap tm_alo;      // two-term A: the A_lo operand
    CUtensorMap tm_a2, tm_alo2, tm_b2, tm_c2;   // the second product (n_split > 0)
    CUtensorMap tm_pool, tm_pool8;               // EPI_KV_POOL: the chunk pool, 128- and 8-row boxes
};

// One product of launch_gemm_pair: C[M, N] = A[M, K] W[N, K]^T + bias (fp32 out),
// A two-term when A_lo is given (as for launch_gemm).
struct GemmProduct {
    const uint16_t* A;
    int64_t lda;
    const uint16_t* A_lo;
    const uint16_t* W;
    int64_t N, K;
    const float* bias;
    float* out;
    int64_t ldo;
};

// ------------------------------------------------------------------ segment projection
struct SegParams {
    int32_t M;           // tokens
    int32_t S;           // segments
    int32_t d_seg;       // 8 or 16
    int32_t num_m, num_g;
    const float* b_seg;  // [S, d_seg]
    uint16_t* y;         // [M, S * d_seg] bf16 (row stride ldy)
    uint16_t* y_lo;      // [M, S * d_seg] remainder y - bf16(y) (row stride ldy), or null
    int64_t ldy;
    unsigned* status;
    uint16_t* kv_out;    // pool variant: assembled cache [M, ld_out]
    int64_t ld_out;
};
// Row map of the pool-reading segment projection: selected chunk i covers
// assembled rows [dst_row[i], dst_row[i] + len[i]), read from pool rows
// starting at src_row[i]; its 128-row tiles are numbered from tile_prefix[i].
struct SegTiles {
    int32_t n_seg;
    int32_t tile_prefix[kMaxSegs + 1];
    int32_t dst_row[kMaxSegs];
    int32_t len[kMaxSegs];
    int64_t src_row[kMaxSegs];
};

// ------------------------------------------------------------------ attention
struct AttnParams {
    const int32_t* chunk_end;    // [N] request-local visible-key end (A0, A3)
    const int32_t* chunk_start;  // [N] request-local chunk start (A3 only)
    int32_t mask_mode;           // cr_mask_mode
    uint16_t* out;           // [N, d_b]
    int32_t d_b;
    int32_t n_heads;
    int32_t n_req;
    int32_t n_items;         // total (request, pair of 128-query tiles) items
    float scale_log2;        // log2(e) / sqrt(d)
    unsigned* status;
    int32_t req_start[kMaxReq + 1];   // cu_seqlens
    int32_t tile_prefix[kMaxReq + 1]; // cumulative items per request
    float* lse;                  // [heads][N] or null: log2-unit log-sum-exp of each row (training)
};

// attention backward (training step)
struct AttnBwdParams {
    const int32_t* chunk_end;     // [N] request-local
    const int32_t* chunk_start;   // [N] request-local
    const float* lse;             // [heads][N] the forward's log-sum-exp (log2 units, scale folded in)
    const float* dvec;            // [heads][N] sum_d dO O
    float* dqkv;                  // [N, 3 d_b] fp32: dQ, dK, dV
    int32_t d_b, n_heads, n_req, n_items, mask_mode;
    float scale_log2;             // log2(e) / sqrt(d)
    float scale;                  // 1 / sqrt(d)
    unsigned* status;
    int32_t req_start[kMaxReq + 1];
    int32_t tile_prefix[kMaxReq + 1];   // cumulative 128-row tiles per request
};

// ------------------------------------------------------------------ training step
struct LossParams {
    int32_t n_req;
    int32_t req_start[kMaxReq + 1];
    float scale[kMaxReq];     // dL/dr factor of each request: 2 / (N_r D_KV n_req)
};
struct AdamWParams {
    float lr, b1, b2, eps, wd, bc1, bc2;
};

// ------------------------------------------------------------------ host helpers
// Target-shape validation shared by every entry point that takes cr_target_dims.
cr_status check_target(const cr_target_dims* t);
unsigned* device_status_ptr();          // per current device, nullptr on failure
int num_sms();                          // SMs of the current device
cr_status cuda_check(cudaError_t e);
bool make_tmap_2d(CUtensorMap* m, const void* base, CUtensorMapDataType dt, uint64_t inner,
                  uint64_t outer, uint64_t row_stride_bytes, uint32_t box_inner,
                  uint32_t box_outer, CUtensorMapSwizzle swz);
inline bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

// Raise a kernel's dynamic shared-memory limit once per device (the first,
// uncaptured call does it, so later calls can be captured into CUDA graphs).
int current_device_index();
// `done` must be a static owned by the caller's kernel-specific code (one per kernel).
// Launch with programmatic dependent launch allowed: the kernel may start (and
// run its prologue) while the previous kernel in the stream finishes; every
// kernel of the library executes griddepcontrol.wait before its first global
// memory access, so it sees all of the previous kernel's writes.
template <typename... P, typename... A>
cr_status launch_pdl(void (*kern)(P...), dim3 grid, dim3 block, size_t smem, cudaStream_t st,
                     A&&... args) {
    cudaLaunchConfig_t cfg = {};
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cuda_check(cudaLaunchKernelEx(&cfg, kern, static_cast<A&&>(args)...));
}

template <typename K>
cr_status ensure_smem_attr(K kern, int bytes, unsigned long long* done) {
    const int d = current_device_index();
    if (d < 0) return CR_ERR_CUDA;
    const unsigned long long bit = 1ull << (d & 63);
    if (__atomic_load_n(done, __ATOMIC_ACQUIRE) & bit) return CR_OK;
    const cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
    if (e != cudaSuccess) return CR_ERR_CUDA;
    __atomic_fetch_or(done, bit, __ATOMIC_ACQ_REL);
    return CR_OK;
}

// Offline preparation: tokens per partial sum of the sigma statistics.
constexpr int64_t kSigmaSlice = 64;

// Launchers (validated arguments).
cr_status launch_gather(const GatherParams& p, cudaStream_t st);
// the pool row of each request token, and per 128-row box and per 8-row group
// its first token's pool row when its rows are one chunk's (else -1)
cr_status launch_src_rows(const GatherParams& p, int64_t* src_row, int64_t* box_src, int64_t* grp_src,
                          cudaStream_t st);
// K segments rotated in place by R_M(dir * (-pos)): dir = +1 canonicalises
// (R_M(q)^{-1}), dir = -1 applies R_M(p).
cr_status launch_canonicalize(void* kv, bool f32, int64_t n, const int32_t* pos, int L, int H, int dh,
                              const float* inv_freq_host, cudaStream_t st, float dir = 1.0f);
cr_status launch_sigma_accumulate(const void* a, const void* b, bool f32, int64_t n, int64_t D,
                                  float* part, double* sumsq, cudaStream_t st);
cr_status launch_sigma_finalize(const double* sumsq, int64_t D, int64_t count, float* sigma,
                                cudaStream_t st);
// A_lo (optional): the second term of a two-term A operand (same shape and
// row stride as A); the product is then (A + A_lo) W^T.
cr_status launch_gemm(const uint16_t* A, int64_t lda, const uint16_t* W, int64_t M, int64_t N,
                      int64_t K, int epi, GemmParams p, void* kv_base, int64_t ld_kv,
                      cudaStream_t st, const uint16_t* A_lo = nullptr);
// The backward's products, C [M, N] fp32 (out = p.out, row stride p.ldo) =, or
// += with EPI_ADD_F32, A' W' where W' [K, N] is stored MN-major (row k of W at
// W + k ldw, N contiguous) and A' [M, K] is A [M, K] K-major (lay LAY_KM = 1) or
// stored [K, M] MN-major (lay LAY_MM = 2), row stride lda.  N a multiple of 64;
// with LAY_MM also M.  No bias.
// scratch (optional, fp32, scratch_bytes long): room for split-K parts; with it
// the product may run as up to 8 k-parts summed in a fixed order afterwards.
// Two fp32 products over the same rows in one launch, so that the tiles of the
// shorter one fill the CTA pairs the other leaves idle.  Falls back to two
// launch_gemm calls where the first product's width is not a multiple of the
// tile width.
cr_status launch_gemm_pair(const GemmProduct& a, const GemmProduct& b, int64_t M, GemmParams p,
                           cudaStream_t st);
cr_status launch_gemm_lay(const uint16_t* A, int64_t lda, int lay, const uint16_t* W, int64_t ldw,
                          int64_t M, int64_t N, int64_t K, int epi, GemmParams p, cudaStream_t st,
                          float* scratch = nullptr, size_t scratch_bytes = 0);
cr_status launch_segproj(const uint16_t* kv, int64_t ld_kv, const uint16_t* wfold, int head_dim,
                         SegParams p, cudaStream_t st);
// The same projection reading the cache tiles straight from the pool (rows
// mapped by `tiles`) and storing each tile, as read, into kv_out [M, D_KV]:
// the stale-cache assembly and stage 1 of the encoder in one pass (bf16).
cr_status launch_segproj_pool(const uint16_t* kv_pool, int64_t n_pool_tokens, uint16_t* kv_out,
                              const uint16_t* wfold, int head_dim, SegParams p,
                              const SegTiles& tiles, cudaStream_t st);
cr_status launch_fold_sigma(const uint16_t* w_seg, const float* sigma, int S, int d_seg,
                            int head_dim, uint16_t* wfold, cudaStream_t st);
cr_status launch_to_bf16(const float* x, int64_t n, uint16_t* y, cudaStream_t st);
// x [rows, cols] fp32 -> out [rows, 2 cols] bf16: each row's hi = rn(x) terms,
// then its lo = rn(x - hi) terms (a two-term A operand for launch_gemm).
cr_status launch_split_bf16(const float* x, int64_t rows, int64_t cols, uint16_t* out,
                            cudaStream_t st);
cr_status launch_rope_table(const int32_t* pos, int64_t n, int half_dim, const float* inv_freq_host,
                            float2* table, cudaStream_t st);
cr_status launch_layernorm(const float* x, const float* add, int64_t ld_add, float* x_out,
                           const float* g, const float* b, float eps, int64_t M, int64_t D,
                           uint16_t* u, cudaStream_t st);
cr_status launch_wait_selftest(unsigned* status, cudaStream_t st);
cr_status launch_chunk_starts(const int32_t* chunk_end, const AttnParams& p, int64_t n_tokens,
                              int32_t* chunk_start, cudaStream_t st);
cr_status launch_attention(const uint16_t* qkv, int64_t n_tokens, int head_dim,
                           const AttnParams& p, cudaStream_t st);

cr_status launch_attention_backward(const uint16_t* qkv, const uint16_t* dO16, const float* dO, const uint16_t* O,
                                    int64_t n_tokens, int head_dim, AttnBwdParams& p, float* dvec, cudaStream_t st);

// training step (cr_train.cu)
// The training head and objective in one pass over the caches: r = W_out y_f +
// b_out - (joint - stale) / sigma_delta from the bf16 stale and joint caches
// [N, D]; writes dz = c_request r (bf16) and the per-request loss, never r or
// the target.  row_scale [N] and part [2 D / 128][N] fp32 are scratch.
cr_status launch_loss_head(const uint16_t* yf, const uint16_t* w_out, const float* b_out,
                           const float* sigma_delta, const uint16_t* stale, const uint16_t* joint, int64_t N,
                           int64_t D, int64_t db, const LossParams& p, uint16_t* dz, float* row_scale,
                           float* part, float* rowsq, float* loss_out, double* per_req, unsigned* status,
                           cudaStream_t st);
size_t colsum_scratch_floats(int64_t rows, int64_t cols);
size_t colsum_counters(int64_t cols);
// Column sums of a contiguous fp32 [rows, cols] matrix (the order of
// launch_colsum) that also write it rounded to bf16 into a16 [rows, cols].
cr_status launch_colsum_bf16(const float* a, int64_t rows, int64_t cols, uint16_t* a16, float* out,
                             float* scratch, unsigned* counters, cudaStream_t st);
cr_status launch_colsum(const void* a, bool bf16, int64_t rows, int64_t cols, int64_t lda, float* out,
                        bool accumulate, float* scratch, unsigned* counters, cudaStream_t st);
cr_status launch_ln_backward(const float* x, const float* gamma, const float* dy, const float* add, float eps,
                             int64_t N, int D, float* dx, float* gprod, cudaStream_t st);
cr_status launch_gelu_backward(float* dg, const float* pre, int64_t n, cudaStream_t st);
cr_status launch_rope_backward(float* dqkv, const float2* table, int64_t N, int db, int hd, cudaStream_t st);
// The W_seg gradient from the grouped dW GEMM's blocks ([S d_h, 128] fp32, the
// rows of segment s carrying its d_seg columns at (s mod (128 / d_seg)) d_seg):
// g [S][d_seg][d_h] = block / sigma_stale (the fold of 1/sigma into W_seg).
cr_status launch_seg_grad(const float* blocks, float* g, int64_t S, int64_t dseg, int64_t dh,
                          const float* sigma, cudaStream_t st);
size_t sqnorm_scratch_doubles();
cr_status launch_clip_adamw(float* p, float* m, float* v, const float* g, uint16_t* pb, int64_t n,
                            const AdamWParams& hp, float max_norm, double* scratch, float* stats,
                            cudaStream_t st);

}  // namespace cr
