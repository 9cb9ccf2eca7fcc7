/*
 * cr.h - C ABI of the GB300 (sm_103a) CacheRepair online repair library.
 *
 * The library repairs a stale multi-chunk KV cache with the lightweight
 * repair network of "CacheRepair: Learning to Repair Cross-Chunk Context in
 * RAG for KV Cache Fusion" (arxiv 2609.35139):
 *
 *     KV_hat = R_theta(KV_stale, D_r)  ~  KV_joint          (Sec. 2.2)
 *
 * in four calls that run back to back on one CUDA stream:
 *
 *   cr_assemble_stale     concatenate canonical chunk caches      (Sec. 4.1)
 *   cr_compress_features  StaleEncoder, token fusion, P_b(s)      (Sec. 4.1)
 *   cr_repair_forward     B Repair Blocks, final LayerNorm        (Sec. 4.1)
 *   cr_apply_residual     KV residual head, in-place residual add,
 *                         optional global RoPE on K               (Sec. 4.1)
 *
 * (cr_assemble_compress runs the first two as one call, with one fewer pass
 * over the cache.)
 *
 * Conventions shared by every call
 * --------------------------------
 * Ownership: the caller owns and allocates every buffer (device memory
 *   unless a parameter says "host").  The library allocates no memory and
 *   keeps no per-call state; scratch lives in a caller workspace of
 *   cr_workspace_bytes() bytes.  Calls on different streams with different
 *   workspaces may run concurrently.
 * Asynchrony: calls enqueue kernels on `stream` (a cudaStream_t; NULL is the
 *   legacy default stream) and return without synchronising.  Host arrays
 *   are read before the call returns.  Nothing is allocated or synchronised,
 *   so a sequence of calls can be captured into a CUDA graph.
 * Layouts: row-major.  A cache row is one token: kv[t, j] with
 *   j = ((layer * 2 + kv) * n_kv_heads + head) * head_dim + d, kv = 0 for K,
 *   D_KV = 2 * n_layers * n_kv_heads * head_dim.  K is canonical (no RoPE,
 *   Sec. 4.1 "Chunk-cache preparation").  Weight matrices are bf16 (uint16
 *   bit patterns) stored [out_features, in_features]; biases, LayerNorm
 *   parameters and sigma vectors are fp32.
 * Alignment: every device pointer must be 16-byte aligned and every row
 *   stride a multiple of 16 bytes (TMA requirement), else CR_ERR_INVALID_ARG.
 * Errors: arguments are validated on the host before anything is enqueued
 *   (CR_ERR_INVALID_ARG, CR_ERR_UNSUPPORTED for shapes the kernels do not
 *   implement); launch failures return CR_ERR_CUDA.  A kernel that detects
 *   a problem on the device (an index out of range, a pipeline wait that
 *   timed out) records it in a device status word instead of trapping; read
 *   it with cr_get_device_status().  Once set, later kernels give up their
 *   waits early, so a bad state never hangs the GPU.
 */
#ifndef CR_H_
#define CR_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum cr_status {
    CR_OK = 0,
    CR_ERR_INVALID_ARG = 1,
    CR_ERR_UNSUPPORTED = 2,
    CR_ERR_CUDA = 3,
    CR_ERR_DEVICE_INDEX = 4,
    CR_ERR_TIMEOUT = 5
} cr_status;

typedef enum cr_dtype { CR_F32 = 0, CR_BF16 = 1 } cr_dtype;

/* Global RoPE on repaired K: none (canonical K out) or R_M(p_t) (Sec. 4.1). */
typedef enum cr_rope_mode { CR_ROPE_NONE = 0, CR_ROPE_GLOBAL = 1 } cr_rope_mode;

/* Attention mask of the Repair Blocks inside one request: the method's
 * block-causal mask (Sec. 4.1) and the attention-topology ablations of
 * App. F.  c(i) is token i's chunk index in the request. */
typedef enum cr_mask_mode {
    CR_MASK_BLOCK_CAUSAL = 0,    /* A0: query i sees key j iff c(j) <= c(i) */
    CR_MASK_TOKEN_CAUSAL = 1,    /* A1: iff j <= i */
    CR_MASK_BIDIRECTIONAL = 2,   /* A2: every key of the request */
    CR_MASK_BLOCK_DIAGONAL = 3   /* A3: iff c(j) == c(i) */
} cr_mask_mode;

/* Output choices of App. F ("Applying the predicted K and V", ablation A5):
 * which cache components receive the predicted correction, and what it is
 * added to. */
typedef enum cr_apply_component { CR_APPLY_K = 1, CR_APPLY_V = 2, CR_APPLY_KV = 3 } cr_apply_component;
typedef enum cr_apply_offset {
    CR_OFFSET_STALE = 0,   /* KV_stale + sigma_Delta z: the method (Sec. 4.1) */
    CR_OFFSET_ZERO = 1     /* sigma_Delta z alone: A5, the head predicts the joint cache */
} cr_apply_offset;

/* Frozen target LLM cache shape (Sec. 4.1: S = 2 L H_KV segments of d_h). */
typedef struct cr_target_dims {
    int32_t n_layers;     /* L_M */
    int32_t n_kv_heads;   /* H_KV */
    int32_t head_dim;     /* d_h: 64 or 128 */
    int32_t d_model;      /* width of the target's token embedding E_M(x_t) */
    int32_t cache_dtype;  /* cr_dtype of the cache and embeddings */
} cr_target_dims;

/* Repairer shape (Sec. 4.1; App. A Table "repair-scales").  d_c is the
 * StaleEncoder/P_tok output width, d_b the backbone width (d_c = d_b in the
 * paper's repairers).  Attention heads are d_b / n_heads wide (32 or 64). */
typedef struct cr_repairer_dims {
    int32_t d_seg;        /* per-segment projection width, 8 or 16 */
    int32_t d_c;
    int32_t d_b;          /* multiple of 128, at most 1024 */
    int32_t n_blocks;     /* B */
    int32_t n_heads;
    int32_t mlp_hidden;   /* MLP width (ratio * d_b) */
    float ln_eps;         /* LayerNorm epsilon */
    float rope_theta;     /* base of the repairer's own RoPE on Q and K */
} cr_repairer_dims;

/* One Repair Block (pre-LN attention + MLP).  Device pointers. */
typedef struct cr_block_weights {
    const float* ln1_g;      /* [d_b] */
    const float* ln1_b;      /* [d_b] */
    const uint16_t* w_qkv;   /* [3 d_b, d_b]: rows 0..d_b-1 Q, then K, then V */
    const float* b_qkv;      /* [3 d_b] */
    const uint16_t* w_o;     /* [d_b, d_b] */
    const float* b_o;        /* [d_b] */
    const float* ln2_g;      /* [d_b] */
    const float* ln2_b;      /* [d_b] */
    const uint16_t* w_fc1;   /* [mlp_hidden, d_b] */
    const float* b_fc1;      /* [mlp_hidden] */
    const uint16_t* w_fc2;   /* [d_b, mlp_hidden] */
    const float* b_fc2;      /* [d_b] */
} cr_block_weights;

/* All repairer parameters (device pointers, except `blocks`, a HOST array of
 * n_blocks entries whose members are device pointers). */
typedef struct cr_weights {
    const uint16_t* w_seg;   /* [S, d_seg, d_h]: segment s's d_h -> d_seg map */
    const float* b_seg;      /* [S, d_seg] */
    const uint16_t* w_map;   /* [d_c, S d_seg] */
    const float* b_map;      /* [d_c] */
    const uint16_t* w_tok;   /* [d_c, d_model]  (P_tok) */
    const float* b_tok;      /* [d_c] */
    const uint16_t* w_fuse;  /* [d_b, 2 d_c]  (F on [s ; P_tok E]) */
    const float* b_fuse;     /* [d_b] */
    const uint16_t* w_rein;  /* [B d_b, d_c]: P_1 .. P_B stacked */
    const float* b_rein;     /* [B d_b] */
    const cr_block_weights* blocks;  /* HOST array [B] */
    const float* lnf_g;      /* [d_b] final LayerNorm */
    const float* lnf_b;      /* [d_b] */
    const uint16_t* w_out;   /* [D_KV, d_b]  KV residual head */
    const float* b_out;      /* [D_KV] */
    const float* sigma_stale;  /* [D_KV] input scale (Sec. 4.2 "Normalization") */
    const float* sigma_delta;  /* [D_KV] residual scale */
} cr_weights;

/* Bytes of scratch workspace the calls need for requests of up to
 * max_tokens assembled tokens (all requests of one call together).
 * Returns 0 if the dimensions are invalid. */
size_t cr_workspace_bytes(const cr_target_dims* target, const cr_repairer_dims* rep,
                          int64_t max_tokens);

/*
 * cr_assemble_stale - concatenate the selected canonical chunk caches of
 * each request in document order into KV^c_stale (Sec. 4.1 "Chunk-cache
 * preparation": with K stored without RoPE, assembly is a pure copy; the
 * method places K at its global position only after repair).
 *
 * kv_pool  [n_pool_tokens, D_KV], emb_pool [n_pool_tokens, d_model]
 *          (cache dtype): independently prefilled chunks back to back.
 * chunk_start [n_pool_chunks] (HOST, int64), chunk_len [n_pool_chunks] (HOST):
 *          pool chunk c occupies rows chunk_start[c] .. + chunk_len[c].
 * chunk_idx (HOST): pool chunk ids of all requests, request r using
 *          chunk_idx[cu_chunks[r] .. cu_chunks[r+1]) in document order.
 * cu_chunks [n_req + 1] (HOST).
 * Outputs (device, caller-sized for max_tokens rows):
 *   kv_out [N, D_KV], emb_out [N, d_model]   stale cache and embeddings
 *   chunk_id  [N] int32  c(t): index of t's chunk within its request
 *   chunk_end [N] int32  exclusive request-local end of t's chunk
 *   pos       [N] int32  p_t: position of t within its request
 *   cu_seqlens_dev [n_req + 1] int32 token offsets of the requests
 *   cu_seqlens_host [n_req + 1] (HOST, written before return)
 * Errors: CR_ERR_INVALID_ARG for an out-of-range or empty chunk, a chunk
 *   outside the pool, an empty request, N > max_tokens, or more than 512
 *   selected chunks / 256 requests in one call.
 */
cr_status cr_assemble_stale(const cr_target_dims* target, const void* kv_pool,
                            const void* emb_pool, int64_t n_pool_tokens,
                            const int64_t* chunk_start, const int32_t* chunk_len,
                            int32_t n_pool_chunks, const int32_t* chunk_idx,
                            const int32_t* cu_chunks, int32_t n_req, void* kv_out,
                            void* emb_out, int64_t max_tokens, int32_t* chunk_id,
                            int32_t* chunk_end, int32_t* pos, int32_t* cu_seqlens_dev,
                            int32_t* cu_seqlens_host, void* stream);

/*
 * cr_compress_features - StaleEncoder and token fusion (Sec. 4.1):
 *   s_t   = W_map [W_seg,s (kv_t,s / sigma_stale,s) + b_seg,s]_s + b_map
 *   h^0_t = F([s_t ; P_tok E_M(x_t)])
 *   r_b   = P_b(s)  for every block b (stale-feature reinjection)
 * kv [N, D_KV], emb [N, d_model] (cache dtype, from cr_assemble_stale).
 * h0_out   [N, d_b] fp32  backbone input h^0.
 * rein_out [N, B d_b] fp32  P_b(s_t) at columns b*d_b .. (b+1)*d_b.
 * Precision: the tensor cores take bf16 operands; the intermediate features
 * (the segment outputs, s and the embedding projection) enter the next
 * linear as two bf16 terms (value = hi + lo, about 16 significant bits), and
 * W_seg / sigma_stale likewise, so that no bf16 rounding of the encoder's
 * features reaches h^0 or the P_b(s), which every block adds into its
 * residual stream.
 * workspace: cr_workspace_bytes(.., max_tokens >= N) bytes, 256-B aligned.
 */
cr_status cr_compress_features(const cr_target_dims* target, const cr_repairer_dims* rep,
                               const cr_weights* w, const void* kv, const void* emb,
                               int64_t n_tokens, float* h0_out, float* rein_out,
                               void* workspace, size_t workspace_bytes, void* stream);

/*
 * cr_assemble_compress - cr_assemble_stale followed by cr_compress_features
 * in one call, with the same arguments and the same results bit for bit
 * (Sec. 4.1, "Chunk-cache preparation" and the StaleEncoder).  For a bf16
 * cache the segment projection reads its cache tiles straight from kv_pool
 * and writes each tile it reads into kv_out, so the assembly costs one read
 * and one write of the cache instead of two reads and a write; fp32 caches
 * take the two-call path.  For a bf16 cache kv_out may be NULL: the assembled
 * cache is then not written at all (cr_apply_residual_pool writes the repaired
 * cache from the pool).  The caller sizes kv_out, emb_out and the
 * workspace (cr_workspace_bytes(.., max_tokens)) for max_tokens rows.
 * Errors: those of the two calls, checked before any launch;
 * CR_ERR_UNSUPPORTED for a NULL kv_out with an fp32 cache.
 */
cr_status cr_assemble_compress(const cr_target_dims* target, const cr_repairer_dims* rep,
                               const cr_weights* w, const void* kv_pool, const void* emb_pool,
                               int64_t n_pool_tokens, const int64_t* chunk_start,
                               const int32_t* chunk_len, int32_t n_pool_chunks,
                               const int32_t* chunk_idx, const int32_t* cu_chunks, int32_t n_req,
                               void* kv_out, void* emb_out, int64_t max_tokens, int32_t* chunk_id,
                               int32_t* chunk_end, int32_t* pos, int32_t* cu_seqlens_dev,
                               int32_t* cu_seqlens_host, float* h0_out, float* rein_out,
                               void* workspace, size_t workspace_bytes, void* stream);

/*
 * cr_repair_forward - the B Repair Blocks and the final LayerNorm (Sec. 4.1):
 *   h^b = RepairBlock_b(h^{b-1} + P_b(s); A, p),   y_f = LN(h^B)
 * with the block-causal mask A_ij = 1[c(j) <= c(i)] inside each request and
 * the repairer's RoPE on Q, K at positions p.
 * h0 [N, d_b] fp32 and rein [N, B d_b] fp32 from cr_compress_features;
 * chunk_end, pos [N] from cr_assemble_stale; cu_seqlens_host [n_req+1] HOST.
 * yf_out [N, d_b] bf16.
 */
cr_status cr_repair_forward(const cr_target_dims* target, const cr_repairer_dims* rep,
                            const cr_weights* w, const float* h0, const float* rein,
                            const int32_t* chunk_end, const int32_t* pos,
                            const int32_t* cu_seqlens_host, int32_t n_req, int64_t n_tokens,
                            uint16_t* yf_out, void* workspace, size_t workspace_bytes,
                            void* stream);

/*
 * cr_repair_forward_masked - cr_repair_forward under any mask of
 * cr_mask_mode: the method's block-causal mask (CR_MASK_BLOCK_CAUSAL, the
 * same computation as cr_repair_forward) or one of the attention-topology
 * ablations A1-A3 of App. F, which change only which keys each query sees.
 * Same arguments and buffers as cr_repair_forward; chunk_end is read for
 * CR_MASK_BLOCK_CAUSAL and CR_MASK_BLOCK_DIAGONAL (for the latter the
 * workspace also receives each token's chunk start).  An unknown mode returns
 * CR_ERR_INVALID_ARG before any launch.
 */
cr_status cr_repair_forward_masked(const cr_target_dims* target, const cr_repairer_dims* rep,
                                   const cr_weights* w, const float* h0, const float* rein,
                                   const int32_t* chunk_end, const int32_t* pos,
                                   const int32_t* cu_seqlens_host, int32_t n_req,
                                   int64_t n_tokens, int32_t mask_mode, uint16_t* yf_out,
                                   void* workspace, size_t workspace_bytes, void* stream);

/*
 * cr_apply_residual - KV residual head and residual add, in place (Sec. 4.1):
 *   z_t = W_out y_f,t + b_out;   kv_t <- round(kv_t + sigma_delta * z_t)
 * and, for CR_ROPE_GLOBAL, K segments rotated by R_M(p_t) (rotate-half pairs
 * (d, d + d_h/2), angle p_t * inv_freq[d]) before the single rounding to the
 * cache dtype (round to nearest even).
 * yf [N, d_b] bf16; kv_inout [N, D_KV] cache dtype; pos [N] device int32;
 * inv_freq_host [head_dim/2] HOST fp32, the target's RoPE frequencies
 * (may be NULL for CR_ROPE_NONE).
 * workspace: NULL, or at least N * head_dim * 4 bytes (16-byte aligned; the
 * cr_workspace_bytes workspace of the other calls is always enough), whose
 * first N * head_dim * 4 bytes are overwritten.  Under CR_ROPE_GLOBAL the call
 * writes R_M's (cos, sin) for every token and rotation pair there once, and
 * the head reads each row's angles from it instead of evaluating them for
 * every K segment of the row; with NULL it evaluates them in the epilogue
 * (the same formula: results agree to one rounding of the cache dtype; more
 * time).  Unused for CR_ROPE_NONE.
 */
cr_status cr_apply_residual(const cr_target_dims* target, const cr_repairer_dims* rep,
                            const cr_weights* w, const uint16_t* yf, int64_t n_tokens,
                            void* kv_inout, const int32_t* pos, const float* inv_freq_host,
                            int32_t rope_mode, void* workspace, size_t workspace_bytes,
                            void* stream);

/*
 * cr_apply_residual_pool - cr_apply_residual for a bf16 cache whose stale rows
 * are read from the chunk pool instead of an assembled cache (Sec. 4.1, KV
 * residual output): for request token t at pool row src(t),
 *   kv_out_t = round(kv_pool[src(t)] + sigma_delta * (W_out y_f,t + b_out))
 * (with R_M on K for CR_ROPE_GLOBAL), the same values bit for bit as
 * cr_assemble_stale followed by cr_apply_residual.  With cr_assemble_compress
 * called without kv_out, the request's cache makes one read in the encoder and
 * one read and one write here, instead of an extra write and read of an
 * assembled copy.  The chunk arguments are those of that call (host arrays,
 * the same checks) and must describe exactly n_tokens rows; kv_out [N, D_KV]
 * receives every row.  workspace: the cr_workspace_bytes(.., >= n_tokens)
 * workspace (its pool-row tables and, under CR_ROPE_GLOBAL, the R_M table are
 * written).  Errors: CR_ERR_UNSUPPORTED for fp32 caches and for D_KV not a
 * multiple of 256; otherwise as the two calls it replaces.
 */
cr_status cr_apply_residual_pool(const cr_target_dims* target, const cr_repairer_dims* rep,
                                 const cr_weights* w, const uint16_t* yf, int64_t n_tokens,
                                 const void* kv_pool, int64_t n_pool_tokens,
                                 const int64_t* chunk_start, const int32_t* chunk_len,
                                 int32_t n_pool_chunks, const int32_t* chunk_idx,
                                 const int32_t* cu_chunks, int32_t n_req, void* kv_out,
                                 const int32_t* pos, const float* inv_freq_host, int32_t rope_mode,
                                 void* workspace, size_t workspace_bytes, void* stream);

/*
 * cr_apply_residual_select - cr_apply_residual under an output choice of
 * App. F.  components: the coordinates that receive the correction
 * (CR_APPLY_K, CR_APPLY_V or both); every other coordinate keeps its stale
 * value bit for bit.  offset: CR_OFFSET_STALE (the method) or CR_OFFSET_ZERO
 * (A5: the repaired value is round(sigma_delta * z)).  keep_chunk_id: NULL, or
 * the chunk map chunk_id [N] device int32 of cr_assemble_stale, in which case
 * the rows of each request's first chunk (chunk_id == 0) keep their stale
 * cache ("keep first chunk").  With CR_ROPE_GLOBAL every K segment leaves
 * rotated by R_M(p_t), repaired or not (an unrepaired K is the stale cache's
 * K, which is rotated to its request position, Sec. 2.2).  A single-component
 * choice needs H_kv * d_h to be a multiple of the head's tile width (256 for
 * bf16 caches, 128 for fp32), else CR_ERR_UNSUPPORTED.  Other arguments as
 * in cr_apply_residual; CR_APPLY_KV with CR_OFFSET_STALE and no kept rows is
 * cr_apply_residual.  Unknown components or offsets: CR_ERR_INVALID_ARG.
 */
cr_status cr_apply_residual_select(const cr_target_dims* target, const cr_repairer_dims* rep,
                                   const cr_weights* w, const uint16_t* yf, int64_t n_tokens,
                                   void* kv_inout, const int32_t* pos, const float* inv_freq_host,
                                   int32_t rope_mode, int32_t components, int32_t offset,
                                   const int32_t* keep_chunk_id, void* workspace,
                                   size_t workspace_bytes, void* stream);

/*
 * cr_rotate_k - K_t <- R_M(p_t) K_t on every K segment, V unchanged, in place:
 * the re-rotation that aligns canonical chunk caches to their request
 * positions in the stale cache (Sec. 2.2; the inverse of
 * cr_canonicalize_chunks).  Assembly followed by this call gives the stale
 * cache KV_stale of independent reuse (the "Stale KV" comparison point).
 * kv_inout [N, D_KV] cache dtype; pos [N] device int32; inv_freq_host
 * [head_dim/2] HOST fp32.  Each rotate-half pair is rotated by p_t f_d and
 * rounded once to the cache dtype.
 */
cr_status cr_rotate_k(const cr_target_dims* target, void* kv_inout, int64_t n_tokens,
                      const int32_t* pos, const float* inv_freq_host, void* stream);

/*
 * cr_apply_residual_paged - the same head and residual add, with the repaired
 * cache written into a paged, layer-major target cache instead of in place:
 * the KV write of the serving integration the paper leaves to future work
 * (Sec. 6 and App. I: pipelining H2D transfer, repair and KV writes; the
 * "KV write" column of the repair-latency table of Sec. 5).  The stale
 * cache is read once and each repaired row is written once, straight from the
 * head GEMM's epilogue, so no separate scatter pass runs.
 *   paged[(2l + kv) * num_slots + slot_mapping[t]][h * d_h + d]
 *       = round(kv_stale[t][((2l + kv) * H_kv + h) * d_h + d] + sigma_delta * z_t)
 * (R_M on K as in cr_apply_residual).  The layout is, per layer and K|V, a
 * [num_slots][H_kv * d_h] array, i.e. [num_blocks][block_size][H_kv][d_h] with
 * slot = block * block_size + offset, planes ordered (layer 0 K, layer 0 V,
 * layer 1 K, ...).  Tokens whose slot is negative are not written (e.g. the
 * tokens after the last complete 16-token block, which the target recomputes
 * with the query); a slot >= num_slots is recorded as a device index error
 * and not written.  Slots of the tokens written must be distinct.
 * yf [N, d_b] bf16; kv_stale [N, D_KV] bf16, read only; pos [N] device int32;
 * slot_mapping [N] device int64; paged_cache [2 L * num_slots * H_kv * d_h]
 * bf16, device; inv_freq_host and workspace as in cr_apply_residual.
 * bf16 caches with H_kv * d_h a multiple of 256 only (else CR_ERR_UNSUPPORTED).
 */
cr_status cr_apply_residual_paged(const cr_target_dims* target, const cr_repairer_dims* rep,
                                  const cr_weights* w, const uint16_t* yf, int64_t n_tokens,
                                  const void* kv_stale, const int32_t* pos,
                                  const float* inv_freq_host, int32_t rope_mode,
                                  const int64_t* slot_mapping, void* paged_cache, int64_t num_slots,
                                  void* workspace, size_t workspace_bytes, void* stream);

/* ---------------------------------------------------------------- offline
 * Preparation that runs once per chunk or once per corpus, not per request.
 *
 * cr_canonicalize_chunks - canonical chunk caches (Sec. 4.1, "Chunk-cache
 * preparation"): each chunk is prefilled alone, and its K is stored without
 * its local rotary encoding,
 *     K^c_t = R_M(q_t)^{-1} K_t,   V^c_t = V_t,
 * q_t the token's position inside its chunk.  In place on kv_inout [N, D_KV]
 * (cache dtype; only K segments are written), pos [N] device int32 = q_t,
 * inv_freq_host [head_dim/2] HOST fp32 (the target's R_M frequencies).  Each
 * rotate-half pair (d, d + d_h/2) of every K segment is rotated by -q_t f_d
 * and rounded once to the cache dtype.
 */
cr_status cr_canonicalize_chunks(const cr_target_dims* target, void* kv_inout, int64_t n_tokens,
                                 const int32_t* pos, const float* inv_freq_host, void* stream);

/*
 * sigma statistics (Sec. 4.2, "Normalization and objective"): one RMS per
 * D_KV coordinate (layer, KV head, K|V, head coordinate) over corpus document
 * tokens; sigma_stale over stale caches, sigma_Delta over the residual targets
 * KV_joint^c - KV_stale^c.  Streamed over the corpus:
 *   cr_sigma_accumulate adds, for every coordinate j, the sum over the call's
 *     n_tokens rows of a[t][j]^2 (or (a[t][j] - b[t][j])^2 when b is not NULL)
 *     to sumsq[j] (device fp64 [D_KV], zeroed by the caller before the first
 *     call); a, b [n_tokens, D_KV] device, cache dtype.  The sum is formed in
 *     a fixed order (fp32 over 64-token slices, fp64 across slices), so equal
 *     inputs give equal bits.  workspace: cr_sigma_workspace_bytes(target,
 *     n_tokens) device bytes, 16-byte aligned.
 *   cr_sigma_finalize writes sigma_out[j] = sqrt(sumsq[j] / count) (fp32
 *     [D_KV], device), count = all rows accumulated.
 */
size_t cr_sigma_workspace_bytes(const cr_target_dims* target, int64_t n_tokens);
cr_status cr_sigma_accumulate(const cr_target_dims* target, const void* a, const void* b,
                              int64_t n_tokens, double* sumsq, void* workspace,
                              size_t workspace_bytes, void* stream);
cr_status cr_sigma_finalize(const cr_target_dims* target, const double* sumsq, int64_t count,
                            float* sigma_out, void* stream);

/* ---------------------------------------------------------------- training
 * One update of the repair network (Sec. 4.2 "Paired cache supervision" and
 * "Normalization and objective"; App. A "Optimization").
 *
 * Parameters live in one flat vector: the trained tensors in this order,
 *   w_seg [S][d_seg][d_h], b_seg [S][d_seg], w_map [d_c][S d_seg], b_map [d_c],
 *   w_tok [d_c][d_model], b_tok [d_c], w_fuse [d_b][2 d_c], b_fuse [d_b],
 *   w_rein [B][d_b][d_c], b_rein [B][d_b],
 *   per block: ln1_g, ln1_b [d_b], w_qkv [3 d_b][d_b], b_qkv [3 d_b],
 *              w_o [d_b][d_b], b_o [d_b], ln2_g, ln2_b [d_b],
 *              w_fc1 [hidden][d_b], b_fc1 [hidden], w_fc2 [d_b][hidden], b_fc2 [d_b],
 *   lnf_g, lnf_b [d_b], w_out [D_KV][d_b], b_out [D_KV],
 * each starting at a multiple of 8 elements (gaps are zero and stay zero).
 * cr_param_layout writes the n_tensors + 1 offsets (the last is the total
 * count) and returns CR_ERR_INVALID_ARG if `max_offsets` is too small; the
 * tensor count is 14 + 12 B.  Row-major [out][in] matrices as elsewhere.
 */
cr_status cr_param_layout(const cr_target_dims* target, const cr_repairer_dims* rep,
                          int64_t* offsets, int32_t max_offsets);

typedef struct cr_adamw {
    float lr;                 /* learning rate of this update */
    float beta1, beta2;       /* (0.9, 0.95) in App. A */
    float eps;                /* 1e-8 */
    float weight_decay;       /* 0.01, decoupled, on every parameter */
    float max_grad_norm;      /* 1: "unit gradient clipping" of the global L2 norm */
    int32_t step;             /* 1-based update count, for the bias corrections */
} cr_adamw;

/* Workspace bytes of cr_train_step for batches of up to max_tokens tokens in
 * total (max_request_tokens, the longest request, must lie in
 * [1, max_tokens]; the fused attention backward needs no per-request
 * scratch); 0 if the dimensions are invalid. */
size_t cr_train_workspace_bytes(const cr_target_dims* target, const cr_repairer_dims* rep,
                                int64_t max_tokens, int64_t max_request_tokens);

/*
 * cr_train_step - forward, objective, backward, clipping and AdamW for one
 * batch of requests (bf16 caches only) under mask_mode, the method's
 * block-causal mask or an attention ablation of App. F (each trained with its
 * own mask there):
 *   L = mean over requests of 1/(N_r D_KV) sum_t || z_t - (KV_joint,t - KV_stale,t) / sigma_Delta ||^2,
 *   g = dL/dtheta over every trained tensor; g <- g min(1, max_norm / (||g|| + 1e-6));
 *   theta <- theta (1 - lr wd) - lr (m / (1 - b1^t)) / (sqrt(v / (1 - b2^t)) + eps)
 * with m, v the AdamW moments.  params [P] fp32 masters (updated in place);
 * params_bf16 [P] their bf16 copies, read by the forward's matrices and
 * rewritten after the update; adam_m, adam_v [P] fp32 (updated); grads [P]
 * fp32, written with the unclipped gradient; sigma_stale, sigma_delta [D_KV]
 * fp32 (fixed statistics, not trained).  kv_stale, kv_joint [N, D_KV] bf16
 * (canonical K), emb [N, d_model] bf16, chunk_end, pos [N] int32 as written by
 * cr_assemble_stale; cu_seqlens_host [n_req + 1] HOST.  stats_out: device
 * fp32 [4] = loss, gradient norm before clipping, clipping coefficient, 0.
 * The forward computes as cr_compress_features + cr_repair_forward (its
 * attention also keeps each row's log-sum-exp); the head and the objective
 * are one GEMM whose epilogue forms the residual from the staged kv_stale and
 * kv_joint tiles and writes dL/dz (bf16) and the rows' squared residuals,
 * never the residual itself; the attention backward is
 * fused (P recomputed tile by tile, no score matrix in memory); the backward's
 * plain matrix products (weight and input gradients) run in the library's
 * tcgen05 GEMM with operands read in their stored layouts (cr_matmul), bf16
 * operands and fp32 accumulation; the W_seg gradient is one grouped product
 * over all segments.  The backward's products need d_c, d_model, mlp_hidden
 * and S d_seg to be multiples of 64 (else CR_ERR_UNSUPPORTED).  All device
 * buffers 16-byte aligned; P = the last offset of cr_param_layout.
 */
cr_status cr_train_step(const cr_target_dims* target, const cr_repairer_dims* rep, float* params,
                        uint16_t* params_bf16, float* adam_m, float* adam_v, float* grads,
                        const float* sigma_stale, const float* sigma_delta, const void* kv_stale,
                        const void* kv_joint, const void* emb, const int32_t* chunk_end,
                        const int32_t* pos, const int32_t* cu_seqlens_host, int32_t n_req,
                        int64_t n_tokens, int32_t mask_mode, const cr_adamw* hp, float* stats_out,
                        void* workspace, size_t workspace_bytes, void* stream);

/* Device status word: out[0] = first error (0 none, 1 wait timeout, 2 device
 * index out of range), out[1] = site, out[2] = block.  Synchronises the
 * device.  cr_clear_device_status() resets it to zero. */
cr_status cr_get_device_status(uint32_t out[3]);
cr_status cr_clear_device_status(void);

const char* cr_status_str(cr_status s);

/* Text of the last CUDA error a call of this thread returned CR_ERR_CUDA for
 * ("no error" if none). */
const char* cr_last_cuda_error(void);

#ifdef __cplusplus
}
#endif
#endif /* CR_H_ */
