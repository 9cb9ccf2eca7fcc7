// C ABI of the repair library (include/cr.h, include/cr_ops.h): host-side
// validation, workspace carving and the launch sequence of each call.
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_runtime.h>
#include <math.h>
#include <algorithm>
#include <memory>
#include <mutex>
#include <vector>
#include <string.h>

#include "cr_internal.h"

// Device status word (first error code, site, block); one copy per device
// that loads the library.  Kernels receive its address as a parameter.
__device__ unsigned g_cr_status[4];

namespace cr {
namespace {

constexpr int kMaxDevices = 64;
std::mutex g_mu;
unsigned* g_status_ptr[kMaxDevices];
int g_sms[kMaxDevices];
PFN_cuTensorMapEncodeTiled_v12000 g_encode = nullptr;

int current_device() {
    int d = -1;
    if (cudaGetDevice(&d) != cudaSuccess || d < 0 || d >= kMaxDevices) return -1;
    return d;
}

size_t align256(size_t x) { return (x + 255) & ~static_cast<size_t>(255); }

struct Dims {
    int64_t L, H, dh, dmodel, S, D;
    bool f32;
    int64_t dseg, dc, db, B, nh, hd, hid;
};

Dims dims_of(const cr_target_dims* t, const cr_repairer_dims* r) {
    Dims d{};
    d.L = t->n_layers;
    d.H = t->n_kv_heads;
    d.dh = t->head_dim;
    d.dmodel = t->d_model;
    d.S = 2 * d.L * d.H;
    d.D = d.S * d.dh;
    d.f32 = t->cache_dtype == CR_F32;
    if (r) {
        d.dseg = r->d_seg;
        d.dc = r->d_c;
        d.db = r->d_b;
        d.B = r->n_blocks;
        d.nh = r->n_heads;
        d.hd = r->n_heads > 0 ? r->d_b / r->n_heads : 0;
        d.hid = r->mlp_hidden;
    }
    return d;
}

}  // namespace

cr_status check_target(const cr_target_dims* t) {
    if (!t) return CR_ERR_INVALID_ARG;
    if (t->n_layers < 1 || t->n_kv_heads < 1 || t->d_model < 8 || (t->d_model % 8) != 0)
        return CR_ERR_INVALID_ARG;
    if (t->cache_dtype != CR_F32 && t->cache_dtype != CR_BF16) return CR_ERR_INVALID_ARG;
    if (t->head_dim != 64 && t->head_dim != 128) return CR_ERR_UNSUPPORTED;
    return CR_OK;
}

namespace {

cr_status check_repairer(const cr_repairer_dims* r) {
    if (!r) return CR_ERR_INVALID_ARG;
    if (r->n_blocks < 0 || r->n_blocks > 64 || r->n_heads < 1 || r->d_c < 16 ||
        r->mlp_hidden < 16 || !(r->ln_eps > 0.0f) || !(r->rope_theta > 0.0f))
        return CR_ERR_INVALID_ARG;
    if (r->d_b % r->n_heads != 0) return CR_ERR_INVALID_ARG;
    if (r->d_seg != 8 && r->d_seg != 16) return CR_ERR_UNSUPPORTED;
    if (r->d_c % 16 != 0 || r->mlp_hidden % 16 != 0) return CR_ERR_UNSUPPORTED;
    if (r->d_b % 128 != 0 || r->d_b > 1024 || r->d_b < 128) return CR_ERR_UNSUPPORTED;
    const int hd = r->d_b / r->n_heads;
    if (hd != 32 && hd != 64) return CR_ERR_UNSUPPORTED;
    return CR_OK;
}

struct WsLayout {
    size_t wfold, kvb, embb, y, se32, se2, x, u, qkv, o, g, rope, kstart, srcrow, boxsrc, grpsrc, total;
};

WsLayout ws_layout(const Dims& d, int64_t n) {
    WsLayout w{};
    size_t off = 0;
    auto take = [&](size_t bytes) {
        const size_t o = off;
        off += align256(bytes);
        return o;
    };
    const size_t N = static_cast<size_t>(n);
    w.wfold = take(static_cast<size_t>(d.S * d.dseg * d.dh) * 2 * 2);   // hi and lo terms
    w.kvb = take(d.f32 ? N * d.D * 2 : 0);
    w.embb = take(d.f32 ? N * d.dmodel * 2 : 0);
    w.y = take(N * d.S * d.dseg * 2 * 2);   // per row [y_hi | y_lo]
    w.se32 = take(N * 2 * d.dc * 4);        // per row [s ; e] fp32
    w.se2 = take(N * 4 * d.dc * 2);         // per row [s_hi e_hi | s_lo e_lo]
    w.x = take(N * d.db * 4);
    w.u = take(N * d.db * 2);
    w.qkv = take(N * 3 * d.db * 2);
    w.o = take(N * d.db * 2);
    w.g = take(N * d.hid * 2);
    w.rope = take(N * (d.hd / 2) * 8);   // repairer RoPE (cos, sin) per token and pair
    w.kstart = take(N * 4);              // chunk start per token (block-diagonal mask)
    w.srcrow = take(N * 8);              // pool row per token (cr_apply_residual_pool)
    w.boxsrc = take((N / 128 + 2) * 8);  // pool row per contiguous 128-row box, or -1
    w.grpsrc = take((N / 128 + 2) * 128);  // pool row per contiguous 8-row group, or -1
    w.total = off;
    return w;
}

template <typename T>
T* at(void* base, size_t off) {
    return reinterpret_cast<T*>(static_cast<uint8_t*>(base) + off);
}

void repairer_inv_freq(float* out, int dim, float theta) {
    for (int i = 0; i < dim / 2; ++i)
        out[i] = static_cast<float>(pow(static_cast<double>(theta), -2.0 * i / dim));
}

bool all_aligned() { return true; }
template <typename P, typename... R>
bool all_aligned(const P* p, R... rest) {
    return p != nullptr && aligned16(p) && all_aligned(rest...);
}
// the same for optional buffers: NULL passes
bool aligned_or_null() { return true; }
template <typename P, typename... R>
bool aligned_or_null(const P* p, R... rest) {
    return (p == nullptr || aligned16(p)) && aligned_or_null(rest...);
}

}  // namespace

namespace {
thread_local cudaError_t t_last_cuda_error = cudaSuccess;
}

cr_status cuda_check(cudaError_t e) {
    if (e == cudaSuccess) return CR_OK;
    t_last_cuda_error = e;
    return CR_ERR_CUDA;
}

int current_device_index() { return current_device(); }

unsigned* device_status_ptr() {
    const int d = current_device();
    if (d < 0) return nullptr;
    std::lock_guard<std::mutex> lk(g_mu);
    if (!g_status_ptr[d]) {
        void* p = nullptr;
        if (cudaGetSymbolAddress(&p, g_cr_status) != cudaSuccess) return nullptr;
        g_status_ptr[d] = static_cast<unsigned*>(p);
    }
    return g_status_ptr[d];
}

int num_sms() {
    const int d = current_device();
    if (d < 0) return 1;
    std::lock_guard<std::mutex> lk(g_mu);
    if (!g_sms[d]) {
        int n = 0;
        if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, d) != cudaSuccess || n < 1)
            n = 1;
        g_sms[d] = n;
    }
    return g_sms[d];
}

bool make_tmap_2d(CUtensorMap* m, const void* base, CUtensorMapDataType dt, uint64_t inner,
                  uint64_t outer, uint64_t row_stride_bytes, uint32_t box_inner,
                  uint32_t box_outer, CUtensorMapSwizzle swz) {
    {
        std::lock_guard<std::mutex> lk(g_mu);
        if (!g_encode) {
            void* fn = nullptr;
            cudaDriverEntryPointQueryResult q;
            if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000,
                                                 cudaEnableDefault, &q) != cudaSuccess ||
                q != cudaDriverEntryPointSuccess || !fn)
                return false;
            g_encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
        }
    }
    if (!aligned16(base) || (row_stride_bytes % 16) != 0 || inner == 0 || outer == 0) return false;
    const cuuint64_t dims[2] = {inner, outer};
    const cuuint64_t strides[1] = {row_stride_bytes};
    const cuuint32_t box[2] = {box_inner, box_outer};
    const cuuint32_t estr[2] = {1, 1};
    return g_encode(m, dt, 2, const_cast<void*>(base), dims, strides, box, estr,
                    CU_TENSOR_MAP_INTERLEAVE_NONE, swz, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                    CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

}  // namespace cr

using namespace cr;

extern "C" {

const char* cr_last_cuda_error(void) {
    return t_last_cuda_error == cudaSuccess ? "no error" : cudaGetErrorString(t_last_cuda_error);
}

const char* cr_status_str(cr_status s) {
    switch (s) {
        case CR_OK: return "ok";
        case CR_ERR_INVALID_ARG: return "invalid argument";
        case CR_ERR_UNSUPPORTED: return "unsupported shape";
        case CR_ERR_CUDA: return "CUDA error";
        case CR_ERR_DEVICE_INDEX: return "device-detected index out of range";
        case CR_ERR_TIMEOUT: return "device pipeline wait timed out";
    }
    return "unknown status";
}

cr_status cr_get_device_status(uint32_t out[3]) {
    if (!out) return CR_ERR_INVALID_ARG;
    unsigned h[4] = {0, 0, 0, 0};
    if (cudaDeviceSynchronize() != cudaSuccess) return CR_ERR_CUDA;
    if (cudaMemcpyFromSymbol(h, g_cr_status, sizeof(h)) != cudaSuccess) return CR_ERR_CUDA;
    out[0] = h[0];
    out[1] = h[1];
    out[2] = h[2];
    if (h[0] == CR_DEV_TIMEOUT) return CR_ERR_TIMEOUT;
    if (h[0] == CR_DEV_INDEX) return CR_ERR_DEVICE_INDEX;
    return CR_OK;
}

cr_status cr_clear_device_status(void) {
    const unsigned z[4] = {0, 0, 0, 0};
    if (cudaMemcpyToSymbol(g_cr_status, z, sizeof(z)) != cudaSuccess) return CR_ERR_CUDA;
    return cudaDeviceSynchronize() == cudaSuccess ? CR_OK : CR_ERR_CUDA;
}

size_t cr_workspace_bytes(const cr_target_dims* target, const cr_repairer_dims* rep,
                          int64_t max_tokens) {
    if (check_target(target) != CR_OK || check_repairer(rep) != CR_OK || max_tokens < 0) return 0;
    return ws_layout(dims_of(target, rep), max_tokens).total;
}

// The gather table of one assembly call from the HOST chunk map (validated):
// every selected chunk's pool rows, output rows and request-local position.
static cr_status build_gather(const Dims& d, const void* kv_pool, const void* emb_pool,
                              int64_t n_pool_tokens, const int64_t* chunk_start,
                              const int32_t* chunk_len, int32_t n_pool_chunks,
                              const int32_t* chunk_idx, const int32_t* cu_chunks, int32_t n_req,
                              void* kv_out, void* emb_out, int64_t max_tokens, int32_t* chunk_id,
                              int32_t* chunk_end, int32_t* pos, int32_t* cu_seqlens_dev,
                              GatherParams* p) {
    if (!chunk_start || !chunk_len || !chunk_idx || !cu_chunks) return CR_ERR_INVALID_ARG;
    if (n_req < 1 || n_req > kMaxReq || n_pool_chunks < 1 || n_pool_tokens < 1)
        return CR_ERR_INVALID_ARG;
    // (the callers say which of the outputs they need)
    if (!all_aligned(kv_pool) || !aligned_or_null(emb_pool, kv_out, emb_out, chunk_id, chunk_end, pos, cu_seqlens_dev))
        return CR_ERR_INVALID_ARG;
    if (cu_chunks[0] != 0) return CR_ERR_INVALID_ARG;
    const int64_t es = d.f32 ? 4 : 2;
    memset(p, 0, sizeof(*p));
    int64_t t = 0;
    int n_seg = 0;
    p->cu_seqlens_host[0] = 0;
    for (int r = 0; r < n_req; ++r) {
        const int a = cu_chunks[r], b = cu_chunks[r + 1];
        if (b <= a || b - a > kMaxSegs) return CR_ERR_INVALID_ARG;
        int64_t local = 0;
        for (int k = a; k < b; ++k) {
            const int c = chunk_idx[k];
            if (c < 0 || c >= n_pool_chunks || n_seg >= kMaxSegs) return CR_ERR_INVALID_ARG;
            const int64_t st = chunk_start[c], ln = chunk_len[c];
            if (ln < 1 || st < 0 || st + ln > n_pool_tokens) return CR_ERR_INVALID_ARG;
            GatherSeg& g = p->seg[n_seg++];
            g.src_row = st;
            g.dst_row = t;
            g.len = static_cast<int32_t>(ln);
            g.chunk_local = k - a;
            g.local_start = static_cast<int32_t>(local);
            local += ln;
            t += ln;
            if (local > INT32_MAX / 2) return CR_ERR_INVALID_ARG;
        }
        p->cu_seqlens_host[r + 1] = static_cast<int32_t>(t);
    }
    if (t > max_tokens || t > INT32_MAX / 2) return CR_ERR_INVALID_ARG;
    p->kv_pool = static_cast<const uint8_t*>(kv_pool);
    p->emb_pool = static_cast<const uint8_t*>(emb_pool);
    p->kv_out = static_cast<uint8_t*>(kv_out);
    p->emb_out = static_cast<uint8_t*>(emb_out);
    p->kv_row_bytes = d.D * es;
    p->emb_row_bytes = d.dmodel * es;
    p->chunk_id = chunk_id;
    p->chunk_end = chunk_end;
    p->pos = pos;
    p->cu_seqlens = cu_seqlens_dev;
    p->n_tokens = t;
    p->n_pool_tokens = n_pool_tokens;
    p->n_seg = n_seg;
    p->n_req = n_req;
    p->status = device_status_ptr();
    return p->status ? CR_OK : CR_ERR_CUDA;
}

cr_status cr_assemble_stale(const cr_target_dims* target, const void* kv_pool,
                            const void* emb_pool, int64_t n_pool_tokens,
                            const int64_t* chunk_start, const int32_t* chunk_len,
                            int32_t n_pool_chunks, const int32_t* chunk_idx,
                            const int32_t* cu_chunks, int32_t n_req, void* kv_out,
                            void* emb_out, int64_t max_tokens, int32_t* chunk_id,
                            int32_t* chunk_end, int32_t* pos, int32_t* cu_seqlens_dev,
                            int32_t* cu_seqlens_host, void* stream) {
    cr_status s = check_target(target);
    if (s != CR_OK) return s;
    if (!cu_seqlens_host) return CR_ERR_INVALID_ARG;
    if (!all_aligned(emb_pool, kv_out, emb_out, chunk_id, chunk_end, pos, cu_seqlens_dev))
        return CR_ERR_INVALID_ARG;
    const Dims d = dims_of(target, nullptr);
    GatherParams* p = new GatherParams();   // ~17 KB: keep it off the caller's stack
    s = build_gather(d, kv_pool, emb_pool, n_pool_tokens, chunk_start, chunk_len, n_pool_chunks,
                     chunk_idx, cu_chunks, n_req, kv_out, emb_out, max_tokens, chunk_id, chunk_end,
                     pos, cu_seqlens_dev, p);
    if (s == CR_OK) {
        for (int r = 0; r <= n_req; ++r) cu_seqlens_host[r] = p->cu_seqlens_host[r];
        s = launch_gather(*p, static_cast<cudaStream_t>(stream));
    }
    delete p;
    return s;
}

static cr_status check_weights_compress(const Dims& d, const cr_weights* w) {
    if (!w) return CR_ERR_INVALID_ARG;
    if (!all_aligned(w->w_seg, w->b_seg, w->w_map, w->b_map, w->w_tok, w->b_tok, w->w_fuse,
                     w->b_fuse, w->sigma_stale))
        return CR_ERR_INVALID_ARG;
    if (d.B > 0 && !all_aligned(w->w_rein, w->b_rein)) return CR_ERR_INVALID_ARG;
    return CR_OK;
}

// Stage 2 and token fusion of the encoder (Sec. 4.1): s = W_map y + b_map,
// e = P_tok E + b_tok, h^0 = F([s ; e]) + b_fuse, and the reinjection terms
// P_b(s) + b_rein.  The encoder's outputs feed the whole residual stream (h^0
// and one P_b(s) per block), so no bf16 rounding is taken there: y comes in
// as two bf16 terms per row ([y_hi | y_lo], from the segment projection); s
// and e are formed in fp32 and split into two terms per row ([s_hi e_hi |
// s_lo e_lo]) for F and the P_b, whose outputs h^0 and P_b(s) stay fp32.
static cr_status compress_stage2(const Dims& d, const cr_weights* w, const uint16_t* y,
                                 const uint16_t* embb, int64_t N, float* h0_out,
                                 float* rein_out, void* workspace, const WsLayout& L,
                                 unsigned* status, cudaStream_t st) {
    cr_status s;
    float* se32 = at<float>(workspace, L.se32);      // [N, 2 d_c] = [s ; P_tok E]
    uint16_t* se2 = at<uint16_t>(workspace, L.se2);  // [N, 4 d_c] two-term bf16
    const int64_t Sd = d.S * d.dseg;
    GemmParams gp{};
    gp.status = status;
    // W_map over [y_hi | y_lo] and P_tok over the embeddings in one launch: the
    // short P_tok tiles fill the CTA pairs the W_map tiles leave idle
    const GemmProduct map{y, 2 * Sd, y + Sd, w->w_map, d.dc, Sd, w->b_map, se32, 2 * d.dc};
    const GemmProduct tok{embb, d.dmodel, nullptr, w->w_tok, d.dc, d.dmodel, w->b_tok, se32 + d.dc,
                          2 * d.dc};
    if ((s = launch_gemm_pair(map, tok, N, gp, st)) != CR_OK) return s;
    if ((s = launch_split_bf16(se32, N, 2 * d.dc, se2, st)) != CR_OK) return s;
    // the fusion F over [s | e] and the reinjection P_b over s, both two-term
    const GemmProduct fuse{se2, 4 * d.dc, se2 + 2 * d.dc, w->w_fuse, d.db, 2 * d.dc, w->b_fuse, h0_out,
                           d.db};
    if (d.B > 0) {
        const GemmProduct rein{se2, 4 * d.dc, se2 + 2 * d.dc, w->w_rein, d.B * d.db, d.dc, w->b_rein,
                               rein_out, d.B * d.db};
        return launch_gemm_pair(fuse, rein, N, gp, st);
    }
    gp.bias = fuse.bias;
    gp.out = fuse.out;
    gp.ldo = fuse.ldo;
    return launch_gemm(fuse.A, fuse.lda, fuse.W, N, fuse.N, fuse.K, EPI_F32, gp, nullptr, 0, st, fuse.A_lo);
}

static SegParams seg_params(const Dims& d, const cr_weights* w, int64_t N, uint16_t* y,
                            unsigned* status) {
    SegParams sp{};
    sp.M = static_cast<int32_t>(N);
    sp.S = static_cast<int32_t>(d.S);
    sp.d_seg = static_cast<int32_t>(d.dseg);
    sp.b_seg = w->b_seg;
    sp.y = y;                     // per row [y_hi | y_lo]
    sp.y_lo = y + d.S * d.dseg;
    sp.ldy = 2 * d.S * d.dseg;
    sp.status = status;
    return sp;
}

// Argument checks shared by the encoder entry points; fills the workspace layout.
static cr_status check_compress(const cr_target_dims* target, const cr_repairer_dims* rep,
                                const cr_weights* w, int64_t max_tokens, float* h0_out,
                                float* rein_out, void* workspace, size_t workspace_bytes,
                                Dims* d, WsLayout* L) {
    cr_status s = check_target(target);
    if (s == CR_OK) s = check_repairer(rep);
    if (s != CR_OK) return s;
    *d = dims_of(target, rep);
    if (max_tokens < 1 || max_tokens > INT32_MAX / 2) return CR_ERR_INVALID_ARG;
    if ((s = check_weights_compress(*d, w)) != CR_OK) return s;
    if (!all_aligned(h0_out, workspace)) return CR_ERR_INVALID_ARG;
    if (d->B > 0 && !all_aligned(rein_out)) return CR_ERR_INVALID_ARG;
    *L = ws_layout(*d, max_tokens);
    if (workspace_bytes < L->total) return CR_ERR_INVALID_ARG;
    return CR_OK;
}

cr_status cr_compress_features(const cr_target_dims* target, const cr_repairer_dims* rep,
                               const cr_weights* w, const void* kv, const void* emb,
                               int64_t n_tokens, float* h0_out, float* rein_out,
                               void* workspace, size_t workspace_bytes, void* stream) {
    Dims d;
    WsLayout L;
    cr_status s = check_compress(target, rep, w, n_tokens, h0_out, rein_out, workspace,
                                 workspace_bytes, &d, &L);
    if (s != CR_OK) return s;
    if (!all_aligned(kv, emb)) return CR_ERR_INVALID_ARG;
    unsigned* status = device_status_ptr();
    if (!status) return CR_ERR_CUDA;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    const int64_t N = n_tokens;

    uint16_t* wfold = at<uint16_t>(workspace, L.wfold);
    if ((s = launch_fold_sigma(w->w_seg, w->sigma_stale, static_cast<int>(d.S),
                               static_cast<int>(d.dseg), static_cast<int>(d.dh), wfold, st)) != CR_OK)
        return s;
    const uint16_t* kvb = static_cast<const uint16_t*>(kv);
    const uint16_t* embb = static_cast<const uint16_t*>(emb);
    if (d.f32) {
        uint16_t* k2 = at<uint16_t>(workspace, L.kvb);
        uint16_t* e2 = at<uint16_t>(workspace, L.embb);
        if ((s = launch_to_bf16(static_cast<const float*>(kv), N * d.D, k2, st)) != CR_OK) return s;
        if ((s = launch_to_bf16(static_cast<const float*>(emb), N * d.dmodel, e2, st)) != CR_OK)
            return s;
        kvb = k2;
        embb = e2;
    }
    uint16_t* y = at<uint16_t>(workspace, L.y);
    const SegParams sp = seg_params(d, w, N, y, status);
    if ((s = launch_segproj(kvb, d.D, wfold, static_cast<int>(d.dh), sp, st)) != CR_OK) return s;
    return compress_stage2(d, w, y, embb, N, h0_out, rein_out, workspace, L, status, st);
}

cr_status cr_assemble_compress(const cr_target_dims* target, const cr_repairer_dims* rep,
                               const cr_weights* w, const void* kv_pool, const void* emb_pool,
                               int64_t n_pool_tokens, const int64_t* chunk_start,
                               const int32_t* chunk_len, int32_t n_pool_chunks,
                               const int32_t* chunk_idx, const int32_t* cu_chunks, int32_t n_req,
                               void* kv_out, void* emb_out, int64_t max_tokens, int32_t* chunk_id,
                               int32_t* chunk_end, int32_t* pos, int32_t* cu_seqlens_dev,
                               int32_t* cu_seqlens_host, float* h0_out, float* rein_out,
                               void* workspace, size_t workspace_bytes, void* stream) {
    Dims d;
    WsLayout L;
    cr_status s = check_compress(target, rep, w, max_tokens, h0_out, rein_out, workspace,
                                 workspace_bytes, &d, &L);
    if (s != CR_OK) return s;
    if (!cu_seqlens_host) return CR_ERR_INVALID_ARG;
    if (!all_aligned(emb_pool, emb_out, chunk_id, chunk_end, pos, cu_seqlens_dev)) return CR_ERR_INVALID_ARG;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    GatherParams* p = new GatherParams();
    s = build_gather(d, kv_pool, emb_pool, n_pool_tokens, chunk_start, chunk_len, n_pool_chunks,
                     chunk_idx, cu_chunks, n_req, kv_out, emb_out, max_tokens, chunk_id, chunk_end,
                     pos, cu_seqlens_dev, p);
    const int64_t N = p->n_tokens;
    // without kv_out (the repaired cache is written from the pool by
    // cr_apply_residual_pool) only the bf16 path applies
    if (s == CR_OK && !kv_out && (d.f32 || n_pool_tokens > INT32_MAX)) s = CR_ERR_UNSUPPORTED;
    if (s == CR_OK && (d.f32 || n_pool_tokens > INT32_MAX)) {
        // fp32 caches go through the bf16 conversion of the two-call form
        for (int r = 0; r <= n_req; ++r) cu_seqlens_host[r] = p->cu_seqlens_host[r];
        s = launch_gather(*p, st);
        delete p;
        if (s != CR_OK) return s;
        return cr_compress_features(target, rep, w, kv_out, emb_out, N, h0_out, rein_out,
                                    workspace, workspace_bytes, stream);
    }
    SegTiles* tl = (s == CR_OK) ? new SegTiles() : nullptr;
    if (s == CR_OK) {
        for (int r = 0; r <= n_req; ++r) cu_seqlens_host[r] = p->cu_seqlens_host[r];
        tl->n_seg = p->n_seg;
        tl->tile_prefix[0] = 0;
        for (int i = 0; i < p->n_seg; ++i) {
            const GatherSeg& g = p->seg[i];
            tl->src_row[i] = g.src_row;
            tl->dst_row[i] = static_cast<int32_t>(g.dst_row);
            tl->len[i] = g.len;
            tl->tile_prefix[i + 1] = tl->tile_prefix[i] + (g.len + 127) / 128;
        }
        // the embeddings and the chunk map here; the cache rows go with the projection
        p->kv_row_bytes = 0;
        s = launch_gather(*p, st);
    }
    unsigned* status = p->status;
    delete p;
    uint16_t* wfold = at<uint16_t>(workspace, L.wfold);
    if (s == CR_OK)
        s = launch_fold_sigma(w->w_seg, w->sigma_stale, static_cast<int>(d.S),
                              static_cast<int>(d.dseg), static_cast<int>(d.dh), wfold, st);
    uint16_t* y = at<uint16_t>(workspace, L.y);
    if (s == CR_OK)
        s = launch_segproj_pool(static_cast<const uint16_t*>(kv_pool), n_pool_tokens,
                                static_cast<uint16_t*>(kv_out), wfold, static_cast<int>(d.dh),
                                seg_params(d, w, N, y, status), *tl, st);
    delete tl;
    if (s != CR_OK) return s;
    return compress_stage2(d, w, y, static_cast<const uint16_t*>(emb_out), N, h0_out, rein_out,
                           workspace, L, status, st);
}

static bool valid_mask_mode(int32_t m) {
    return m == CR_MASK_BLOCK_CAUSAL || m == CR_MASK_TOKEN_CAUSAL || m == CR_MASK_BIDIRECTIONAL ||
           m == CR_MASK_BLOCK_DIAGONAL;
}

static cr_status attn_params(const Dims& d, int32_t mask_mode, const int32_t* chunk_end,
                             const int32_t* chunk_start, const int32_t* cu_seqlens_host, int n_req,
                             int64_t N, uint16_t* out, unsigned* status, AttnParams* p) {
    if (!cu_seqlens_host || n_req < 1 || n_req > kMaxReq) return CR_ERR_INVALID_ARG;
    if (!valid_mask_mode(mask_mode)) return CR_ERR_INVALID_ARG;
    if ((mask_mode == CR_MASK_BLOCK_CAUSAL || mask_mode == CR_MASK_BLOCK_DIAGONAL) &&
        !all_aligned(chunk_end))
        return CR_ERR_INVALID_ARG;
    if (mask_mode == CR_MASK_BLOCK_DIAGONAL && !all_aligned(chunk_start)) return CR_ERR_INVALID_ARG;
    if (cu_seqlens_host[0] != 0 || cu_seqlens_host[n_req] != N) return CR_ERR_INVALID_ARG;
    memset(p, 0, sizeof(*p));
    int items = 0;
    for (int r = 0; r < n_req; ++r) {
        const int len = cu_seqlens_host[r + 1] - cu_seqlens_host[r];
        if (len < 1) return CR_ERR_INVALID_ARG;
        p->req_start[r] = cu_seqlens_host[r];
        p->tile_prefix[r] = items;
        items += (len + 255) / 256;       // pairs of 128-query tiles
    }
    p->req_start[n_req] = cu_seqlens_host[n_req];
    p->tile_prefix[n_req] = items;
    p->chunk_end = chunk_end;
    p->chunk_start = chunk_start;
    p->mask_mode = mask_mode;
    p->out = out;
    p->d_b = static_cast<int32_t>(d.db);
    p->n_heads = static_cast<int32_t>(d.nh);
    p->n_req = n_req;
    p->n_items = items;
    p->scale_log2 = static_cast<float>(1.4426950408889634 / sqrt(static_cast<double>(d.hd)));
    p->status = status;
    return CR_OK;
}

cr_status cr_repair_forward(const cr_target_dims* target, const cr_repairer_dims* rep,
                            const cr_weights* w, const float* h0, const float* rein,
                            const int32_t* chunk_end, const int32_t* pos,
                            const int32_t* cu_seqlens_host, int32_t n_req, int64_t n_tokens,
                            uint16_t* yf_out, void* workspace, size_t workspace_bytes,
                            void* stream) {
    return cr_repair_forward_masked(target, rep, w, h0, rein, chunk_end, pos, cu_seqlens_host,
                                    n_req, n_tokens, CR_MASK_BLOCK_CAUSAL, yf_out, workspace,
                                    workspace_bytes, stream);
}

cr_status cr_repair_forward_masked(const cr_target_dims* target, const cr_repairer_dims* rep,
                                   const cr_weights* w, const float* h0, const float* rein,
                                   const int32_t* chunk_end, const int32_t* pos,
                                   const int32_t* cu_seqlens_host, int32_t n_req,
                                   int64_t n_tokens, int32_t mask_mode, uint16_t* yf_out,
                                   void* workspace, size_t workspace_bytes, void* stream) {
    cr_status s = check_target(target);
    if (s == CR_OK) s = check_repairer(rep);
    if (s != CR_OK) return s;
    const Dims d = dims_of(target, rep);
    if (!w || n_tokens < 1 || n_tokens > INT32_MAX / 2) return CR_ERR_INVALID_ARG;
    if (!all_aligned(h0, chunk_end, pos, yf_out, workspace, w->lnf_g, w->lnf_b))
        return CR_ERR_INVALID_ARG;
    if (!valid_mask_mode(mask_mode)) return CR_ERR_INVALID_ARG;
    if (d.B > 0 && (!w->blocks || !all_aligned(rein))) return CR_ERR_INVALID_ARG;
    for (int b = 0; b < d.B; ++b) {
        const cr_block_weights& k = w->blocks[b];
        if (!all_aligned(k.ln1_g, k.ln1_b, k.w_qkv, k.b_qkv, k.w_o, k.b_o, k.ln2_g, k.ln2_b,
                         k.w_fc1, k.b_fc1, k.w_fc2, k.b_fc2))
            return CR_ERR_INVALID_ARG;
    }
    const WsLayout L = ws_layout(d, n_tokens);
    if (workspace_bytes < L.total) return CR_ERR_INVALID_ARG;
    const int64_t N = n_tokens;
    float* x = at<float>(workspace, L.x);
    uint16_t* u = at<uint16_t>(workspace, L.u);
    uint16_t* qkv = at<uint16_t>(workspace, L.qkv);
    uint16_t* o = at<uint16_t>(workspace, L.o);
    uint16_t* g = at<uint16_t>(workspace, L.g);
    int32_t* kstart = at<int32_t>(workspace, L.kstart);
    AttnParams* ap = new AttnParams();
    s = attn_params(d, mask_mode, chunk_end, kstart, cu_seqlens_host, n_req, N, o, nullptr, ap);
    unsigned* status = (s == CR_OK) ? device_status_ptr() : nullptr;
    if (s == CR_OK && !status) s = CR_ERR_CUDA;
    if (s != CR_OK) {
        delete ap;
        return s;
    }
    ap->status = status;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    // the block-diagonal mask also needs each token's chunk start: once per forward
    if (mask_mode == CR_MASK_BLOCK_DIAGONAL && d.B > 0) {
        s = launch_chunk_starts(chunk_end, *ap, N, kstart, st);
        if (s != CR_OK) {
            delete ap;
            return s;
        }
    }
    GemmParams gq{};
    gq.status = status;
    gq.pos = pos;
    gq.rope_dim = static_cast<int32_t>(d.hd);
    gq.rope_cols = static_cast<int32_t>(2 * d.db);
    repairer_inv_freq(gq.inv_freq, static_cast<int>(d.hd), rep->rope_theta);
    // positions are the same for every block: one (cos, sin) table per forward
    float2* rope = at<float2>(workspace, L.rope);
    if (d.B > 0) {
        s = launch_rope_table(pos, N, static_cast<int>(d.hd / 2), gq.inv_freq, rope, st);
        if (s != CR_OK) {
            delete ap;
            return s;
        }
        gq.rope_table = rope;
    }
    GemmParams gr{};
    gr.status = status;
    for (int b = 0; b < d.B && s == CR_OK; ++b) {
        const cr_block_weights& k = w->blocks[b];
        // x = h^{b-1} + P_b(s);  u = LN1(x)
        s = launch_layernorm(b == 0 ? h0 : x, rein + b * d.db, d.B * d.db, x, k.ln1_g, k.ln1_b,
                             rep->ln_eps, N, d.db, u, st);
        if (s != CR_OK) break;
        gq.bias = k.b_qkv;
        gq.out = qkv;
        gq.ldo = 3 * d.db;
        s = launch_gemm(u, d.db, k.w_qkv, N, 3 * d.db, d.db, EPI_QKV_ROPE, gq, nullptr, 0, st);
        if (s != CR_OK) break;
        s = launch_attention(qkv, N, static_cast<int>(d.hd), *ap, st);
        if (s != CR_OK) break;
        gr.bias = k.b_o;
        gr.out = x;
        gr.ldo = d.db;
        s = launch_gemm(o, d.db, k.w_o, N, d.db, d.db, EPI_ADD_F32, gr, nullptr, 0, st);
        if (s != CR_OK) break;
        s = launch_layernorm(x, nullptr, 0, x, k.ln2_g, k.ln2_b, rep->ln_eps, N, d.db, u, st);
        if (s != CR_OK) break;
        gr.bias = k.b_fc1;
        gr.out = g;
        gr.ldo = d.hid;
        s = launch_gemm(u, d.db, k.w_fc1, N, d.hid, d.db, EPI_GELU_BF16, gr, nullptr, 0, st);
        if (s != CR_OK) break;
        gr.bias = k.b_fc2;
        gr.out = x;
        gr.ldo = d.db;
        s = launch_gemm(g, d.hid, k.w_fc2, N, d.db, d.hid, EPI_ADD_F32, gr, nullptr, 0, st);
    }
    delete ap;
    if (s != CR_OK) return s;
    return launch_layernorm(d.B > 0 ? x : h0, nullptr, 0, nullptr, w->lnf_g, w->lnf_b,
                            rep->ln_eps, N, d.db, yf_out, st);
}

cr_status cr_apply_residual(const cr_target_dims* target, const cr_repairer_dims* rep,
                            const cr_weights* w, const uint16_t* yf, int64_t n_tokens,
                            void* kv_inout, const int32_t* pos, const float* inv_freq_host,
                            int32_t rope_mode, void* workspace, size_t workspace_bytes,
                            void* stream) {
    return cr_apply_residual_select(target, rep, w, yf, n_tokens, kv_inout, pos, inv_freq_host,
                                    rope_mode, CR_APPLY_KV, CR_OFFSET_STALE, nullptr, workspace,
                                    workspace_bytes, stream);
}

// R_M's (cos, sin) for every token and pair index (angle-major, entry q N + t),
// written once per call into the caller's workspace, so that the head's
// epilogue reads each row's angles instead of evaluating them for every K
// segment.  Without a workspace the epilogue evaluates them itself.
static cr_status target_rope_table(const Dims& d, const int32_t* pos, int64_t n_tokens,
                                   const float* inv_freq_host, void* workspace,
                                   size_t workspace_bytes, GemmParams* gp, cudaStream_t st) {
    if (!workspace) return CR_OK;
    const size_t bytes = static_cast<size_t>(n_tokens) * static_cast<size_t>(d.dh / 2) * 8;
    if (!all_aligned(workspace) || workspace_bytes < bytes) return CR_ERR_INVALID_ARG;
    float2* table = static_cast<float2*>(workspace);
    const cr_status s = launch_rope_table(pos, n_tokens, static_cast<int>(d.dh / 2), inv_freq_host, table, st);
    if (s == CR_OK) gp->rope_table = table;
    return s;
}

cr_status cr_apply_residual_select(const cr_target_dims* target, const cr_repairer_dims* rep,
                                   const cr_weights* w, const uint16_t* yf, int64_t n_tokens,
                                   void* kv_inout, const int32_t* pos, const float* inv_freq_host,
                                   int32_t rope_mode, int32_t components, int32_t offset,
                                   const int32_t* keep_chunk_id, void* workspace,
                                   size_t workspace_bytes, void* stream) {
    cr_status s = check_target(target);
    if (s == CR_OK) s = check_repairer(rep);
    if (s != CR_OK) return s;
    const Dims d = dims_of(target, rep);
    if (!w || n_tokens < 1 || n_tokens > INT32_MAX / 2) return CR_ERR_INVALID_ARG;
    if (rope_mode != CR_ROPE_NONE && rope_mode != CR_ROPE_GLOBAL) return CR_ERR_INVALID_ARG;
    if (!all_aligned(yf, kv_inout, pos, w->w_out, w->b_out, w->sigma_delta))
        return CR_ERR_INVALID_ARG;
    if (rope_mode == CR_ROPE_GLOBAL && !inv_freq_host) return CR_ERR_INVALID_ARG;
    if (components != CR_APPLY_K && components != CR_APPLY_V && components != CR_APPLY_KV)
        return CR_ERR_INVALID_ARG;
    if (offset != CR_OFFSET_STALE && offset != CR_OFFSET_ZERO) return CR_ERR_INVALID_ARG;
    if (keep_chunk_id && !all_aligned(keep_chunk_id)) return CR_ERR_INVALID_ARG;
    const int bn = d.f32 ? 128 : 256;
    if (d.D % bn != 0) return CR_ERR_UNSUPPORTED;
    const int64_t plane = static_cast<int64_t>(d.H) * d.dh;   // one (layer, K|V) block
    if (components != CR_APPLY_KV && plane % bn != 0) return CR_ERR_UNSUPPORTED;
    unsigned* status = device_status_ptr();
    if (!status) return CR_ERR_CUDA;
    GemmParams gp{};
    gp.status = status;
    gp.bias = w->b_out;
    gp.sigma = w->sigma_delta;
    gp.pos = pos;
    gp.rope_dim = static_cast<int32_t>(d.dh);
    gp.rope_on = rope_mode == CR_ROPE_GLOBAL ? 1 : 0;
    gp.n_kv_heads = static_cast<int32_t>(d.H);
    if (gp.rope_on)
        for (int i = 0; i < d.dh / 2; ++i) gp.inv_freq[i] = inv_freq_host[i];
    if (components != CR_APPLY_KV) {
        gp.col_block = static_cast<int32_t>(plane);
        gp.col_phase = components == CR_APPLY_K ? 0 : 1;
    }
    gp.kv_zero = offset == CR_OFFSET_ZERO ? 1 : 0;
    gp.keep_chunk = keep_chunk_id;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    if (gp.rope_on && components != CR_APPLY_V &&
        (s = target_rope_table(d, pos, n_tokens, inv_freq_host, workspace, workspace_bytes, &gp, st)) != CR_OK)
        return s;
    s = launch_gemm(yf, d.db, w->w_out, n_tokens, d.D, d.db, d.f32 ? EPI_KV_F32 : EPI_KV_BF16, gp,
                    kv_inout, d.D, st);
    // V-only under the target's R_M: the K segments the head did not visit are
    // still rotated to their request positions
    if (s == CR_OK && gp.rope_on && components == CR_APPLY_V)
        s = launch_canonicalize(kv_inout, d.f32, n_tokens, pos, static_cast<int>(d.L),
                                static_cast<int>(d.H), static_cast<int>(d.dh), inv_freq_host, st,
                                -1.0f);
    return s;
}

cr_status cr_apply_residual_pool(const cr_target_dims* target, const cr_repairer_dims* rep,
                                 const cr_weights* w, const uint16_t* yf, int64_t n_tokens,
                                 const void* kv_pool, int64_t n_pool_tokens,
                                 const int64_t* chunk_start, const int32_t* chunk_len,
                                 int32_t n_pool_chunks, const int32_t* chunk_idx,
                                 const int32_t* cu_chunks, int32_t n_req, void* kv_out,
                                 const int32_t* pos, const float* inv_freq_host, int32_t rope_mode,
                                 void* workspace, size_t workspace_bytes, void* stream) {
    cr_status s = check_target(target);
    if (s == CR_OK) s = check_repairer(rep);
    if (s != CR_OK) return s;
    const Dims d = dims_of(target, rep);
    if (d.f32) return CR_ERR_UNSUPPORTED;   // bf16 caches (the fused front's path)
    if (!w || !kv_pool || !kv_out || !workspace || n_tokens < 1 || n_tokens > INT32_MAX / 2 ||
        n_pool_tokens < 1 || n_pool_tokens > INT32_MAX)
        return CR_ERR_INVALID_ARG;
    if (rope_mode != CR_ROPE_NONE && rope_mode != CR_ROPE_GLOBAL) return CR_ERR_INVALID_ARG;
    if (rope_mode == CR_ROPE_GLOBAL && !inv_freq_host) return CR_ERR_INVALID_ARG;
    if (!all_aligned(yf, kv_pool, kv_out, pos, workspace, w->w_out, w->b_out, w->sigma_delta))
        return CR_ERR_INVALID_ARG;
    if (d.D % 256 != 0) return CR_ERR_UNSUPPORTED;
    const WsLayout L = ws_layout(d, n_tokens);
    if (workspace_bytes < L.total) return CR_ERR_INVALID_ARG;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    GatherParams* gpl = new GatherParams();
    s = build_gather(d, kv_pool, nullptr, n_pool_tokens, chunk_start, chunk_len, n_pool_chunks, chunk_idx,
                     cu_chunks, n_req, nullptr, nullptr, n_tokens, nullptr, nullptr, nullptr, nullptr, gpl);
    if (s == CR_OK && gpl->n_tokens != n_tokens) s = CR_ERR_INVALID_ARG;
    int64_t* src_row = at<int64_t>(workspace, L.srcrow);
    int64_t* box_src = at<int64_t>(workspace, L.boxsrc);
    int64_t* grp_src = at<int64_t>(workspace, L.grpsrc);
    if (s == CR_OK) s = launch_src_rows(*gpl, src_row, box_src, grp_src, st);
    unsigned* status = gpl->status;
    delete gpl;
    if (s != CR_OK) return s;
    GemmParams gp{};
    gp.status = status;
    gp.bias = w->b_out;
    gp.sigma = w->sigma_delta;
    gp.pos = pos;
    gp.rope_dim = static_cast<int32_t>(d.dh);
    gp.rope_on = rope_mode == CR_ROPE_GLOBAL ? 1 : 0;
    gp.n_kv_heads = static_cast<int32_t>(d.H);
    if (gp.rope_on) {
        for (int i = 0; i < d.dh / 2; ++i) gp.inv_freq[i] = inv_freq_host[i];
        // (the R_M table sits at the front of the workspace, clear of the row tables)
        if ((s = target_rope_table(d, pos, n_tokens, inv_freq_host, workspace, workspace_bytes, &gp, st)) != CR_OK)
            return s;
    }
    gp.kv_pool = static_cast<const uint16_t*>(kv_pool);
    gp.src_row = src_row;
    gp.box_src = box_src;
    gp.grp_src = grp_src;
    if (!make_tmap_2d(&gp.tm_pool, kv_pool, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, d.D, n_pool_tokens, d.D * 2, 64,
                      128, CU_TENSOR_MAP_SWIZZLE_128B) ||
        !make_tmap_2d(&gp.tm_pool8, kv_pool, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, d.D, n_pool_tokens, d.D * 2, 64,
                      8, CU_TENSOR_MAP_SWIZZLE_128B))
        return CR_ERR_INVALID_ARG;
    return launch_gemm(yf, d.db, w->w_out, n_tokens, d.D, d.db, EPI_KV_POOL, gp, kv_out, d.D, st);
}

cr_status cr_rotate_k(const cr_target_dims* target, void* kv_inout, int64_t n_tokens,
                      const int32_t* pos, const float* inv_freq_host, void* stream) {
    const cr_status s = check_target(target);
    if (s != CR_OK) return s;
    if (n_tokens < 1 || !inv_freq_host || !all_aligned(kv_inout, pos)) return CR_ERR_INVALID_ARG;
    const Dims d = dims_of(target, nullptr);
    if (n_tokens > INT64_MAX / (d.D * 4)) return CR_ERR_INVALID_ARG;
    return launch_canonicalize(kv_inout, d.f32, n_tokens, pos, static_cast<int>(d.L),
                               static_cast<int>(d.H), static_cast<int>(d.dh), inv_freq_host,
                               static_cast<cudaStream_t>(stream), -1.0f);
}

cr_status cr_apply_residual_paged(const cr_target_dims* target, const cr_repairer_dims* rep,
                                  const cr_weights* w, const uint16_t* yf, int64_t n_tokens,
                                  const void* kv_stale, const int32_t* pos,
                                  const float* inv_freq_host, int32_t rope_mode,
                                  const int64_t* slot_mapping, void* paged_cache, int64_t num_slots,
                                  void* workspace, size_t workspace_bytes, void* stream) {
    cr_status s = check_target(target);
    if (s == CR_OK) s = check_repairer(rep);
    if (s != CR_OK) return s;
    const Dims d = dims_of(target, rep);
    if (!w || n_tokens < 1 || n_tokens > INT32_MAX / 2 || num_slots < 1) return CR_ERR_INVALID_ARG;
    if (rope_mode != CR_ROPE_NONE && rope_mode != CR_ROPE_GLOBAL) return CR_ERR_INVALID_ARG;
    if (!all_aligned(yf, kv_stale, pos, slot_mapping, paged_cache, w->w_out, w->b_out,
                     w->sigma_delta))
        return CR_ERR_INVALID_ARG;
    if (rope_mode == CR_ROPE_GLOBAL && !inv_freq_host) return CR_ERR_INVALID_ARG;
    const int64_t plane = static_cast<int64_t>(d.H) * d.dh;   // one (layer, K|V) row
    if (d.f32 || plane % 256 != 0 || d.D % 256 != 0) return CR_ERR_UNSUPPORTED;
    if (num_slots > INT64_MAX / (2 * static_cast<int64_t>(d.L) * plane)) return CR_ERR_INVALID_ARG;
    unsigned* status = device_status_ptr();
    if (!status) return CR_ERR_CUDA;
    GemmParams gp{};
    gp.status = status;
    gp.bias = w->b_out;
    gp.sigma = w->sigma_delta;
    gp.pos = pos;
    gp.rope_dim = static_cast<int32_t>(d.dh);
    gp.rope_on = rope_mode == CR_ROPE_GLOBAL ? 1 : 0;
    gp.n_kv_heads = static_cast<int32_t>(d.H);
    if (gp.rope_on)
        for (int i = 0; i < d.dh / 2; ++i) gp.inv_freq[i] = inv_freq_host[i];
    gp.slot = slot_mapping;
    gp.paged = static_cast<uint16_t*>(paged_cache);
    gp.num_slots = num_slots;
    gp.seg_width = static_cast<int32_t>(plane);
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    if (gp.rope_on &&
        (s = target_rope_table(d, pos, n_tokens, inv_freq_host, workspace, workspace_bytes, &gp, st)) != CR_OK)
        return s;
    // the stale tile is read through the same tensor map as the in-place update
    return launch_gemm(yf, d.db, w->w_out, n_tokens, d.D, d.db, EPI_KV_PAGED, gp,
                       const_cast<void*>(kv_stale), d.D, st);
}

// ------------------------------------------------------------------ offline preparation
cr_status cr_canonicalize_chunks(const cr_target_dims* target, void* kv_inout, int64_t n_tokens,
                                 const int32_t* pos, const float* inv_freq_host, void* stream) {
    const cr_status s = check_target(target);
    if (s != CR_OK) return s;
    if (n_tokens < 1 || !inv_freq_host || !all_aligned(kv_inout, pos)) return CR_ERR_INVALID_ARG;
    const Dims d = dims_of(target, nullptr);
    if (n_tokens > INT64_MAX / (d.D * 4)) return CR_ERR_INVALID_ARG;
    return launch_canonicalize(kv_inout, d.f32, n_tokens, pos, static_cast<int>(d.L),
                               static_cast<int>(d.H), static_cast<int>(d.dh), inv_freq_host,
                               static_cast<cudaStream_t>(stream));
}

size_t cr_sigma_workspace_bytes(const cr_target_dims* target, int64_t n_tokens) {
    if (check_target(target) != CR_OK || n_tokens < 1) return 0;
    const Dims d = dims_of(target, nullptr);
    const int64_t slices = (n_tokens + kSigmaSlice - 1) / kSigmaSlice;
    return align256(static_cast<size_t>(slices) * static_cast<size_t>(d.D) * sizeof(float));
}

cr_status cr_sigma_accumulate(const cr_target_dims* target, const void* a, const void* b,
                              int64_t n_tokens, double* sumsq, void* workspace,
                              size_t workspace_bytes, void* stream) {
    const cr_status s = check_target(target);
    if (s != CR_OK) return s;
    if (n_tokens < 1 || !all_aligned(a, sumsq, workspace) || (b && !aligned16(b)))
        return CR_ERR_INVALID_ARG;
    if (workspace_bytes < cr_sigma_workspace_bytes(target, n_tokens)) return CR_ERR_INVALID_ARG;
    const Dims d = dims_of(target, nullptr);
    return launch_sigma_accumulate(a, b, d.f32, n_tokens, d.D, static_cast<float*>(workspace), sumsq,
                                   static_cast<cudaStream_t>(stream));
}

cr_status cr_sigma_finalize(const cr_target_dims* target, const double* sumsq, int64_t count,
                            float* sigma_out, void* stream) {
    const cr_status s = check_target(target);
    if (s != CR_OK) return s;
    if (count < 1 || !all_aligned(sumsq, sigma_out)) return CR_ERR_INVALID_ARG;
    const Dims d = dims_of(target, nullptr);
    return launch_sigma_finalize(sumsq, d.D, count, sigma_out, static_cast<cudaStream_t>(stream));
}

// ------------------------------------------------------------------ cr_ops.h
cr_status cr_linear(const uint16_t* A, int64_t lda, const uint16_t* W, const float* bias,
                    int64_t M, int64_t N, int64_t K, void* out, int64_t ldo, int32_t epi,
                    void* stream) {
    if (M < 1 || N < 1 || K < 8 || (K % 8) != 0 || (N % 16) != 0 || lda < K || ldo < N)
        return CR_ERR_INVALID_ARG;
    if (M > INT32_MAX / 2 || N > INT32_MAX / 2 || K > INT32_MAX / 2) return CR_ERR_INVALID_ARG;
    if (epi < CR_EPI_BF16 || epi > CR_EPI_F32) return CR_ERR_INVALID_ARG;
    if (!all_aligned(A, W, out) || (bias && !aligned16(bias))) return CR_ERR_INVALID_ARG;
    const int64_t es = (epi == CR_EPI_ADD_F32 || epi == CR_EPI_F32) ? 4 : 2;
    if ((lda * 2) % 16 != 0 || (ldo * es) % 16 != 0) return CR_ERR_INVALID_ARG;
    unsigned* status = device_status_ptr();
    if (!status) return CR_ERR_CUDA;
    GemmParams gp{};
    gp.status = status;
    gp.bias = bias;
    gp.out = out;
    gp.ldo = ldo;
    static const int map[4] = {EPI_BF16, EPI_GELU_BF16, EPI_ADD_F32, EPI_F32};
    return launch_gemm(A, lda, W, M, N, K, map[epi], gp, nullptr, 0,
                       static_cast<cudaStream_t>(stream));
}

cr_status cr_matmul(const uint16_t* A, int64_t lda, int32_t a_trans, const uint16_t* B, int64_t ldb,
                    int64_t M, int64_t N, int64_t K, float* C, int64_t ldc, int32_t accumulate,
                    void* workspace, size_t workspace_bytes, void* stream) {
    if (M < 1 || N < 1 || K < 1 || M > INT32_MAX / 2 || N > INT32_MAX / 2 || K > INT32_MAX / 2)
        return CR_ERR_INVALID_ARG;
    if (workspace && !all_aligned(workspace)) return CR_ERR_INVALID_ARG;
    if (!all_aligned(A, B, C) || (lda % 8) != 0 || (ldb % 8) != 0 || (ldc % 4) != 0 || ldb < N ||
        ldc < N || lda < (a_trans ? M : K))
        return CR_ERR_INVALID_ARG;
    if ((N % 64) != 0 || (a_trans && (M % 64) != 0)) return CR_ERR_UNSUPPORTED;
    unsigned* status = device_status_ptr();
    if (!status) return CR_ERR_CUDA;
    GemmParams gp{};
    gp.status = status;
    gp.out = C;
    gp.ldo = ldc;
    return launch_gemm_lay(A, lda, a_trans ? LAY_MM : LAY_KM, B, ldb, M, N, K,
                           accumulate ? EPI_ADD_F32 : EPI_F32, gp, static_cast<cudaStream_t>(stream),
                           static_cast<float*>(workspace), workspace ? workspace_bytes : 0);
}

cr_status cr_layernorm(const float* x, const float* add, int64_t ld_add, float* x_out,
                       const float* gamma, const float* beta, float eps, int64_t M, int64_t D,
                       uint16_t* u, void* stream) {
    if (M < 1 || D < 128 || D > 1024 || (D % 128) != 0 || !(eps > 0.0f)) return CR_ERR_INVALID_ARG;
    if (!all_aligned(x, gamma, beta, u)) return CR_ERR_INVALID_ARG;
    if (add && (!all_aligned(add, x_out) || ld_add < D || (ld_add % 4) != 0))
        return CR_ERR_INVALID_ARG;
    return launch_layernorm(x, add, ld_add, x_out, gamma, beta, eps, M, D, u,
                            static_cast<cudaStream_t>(stream));
}

cr_status cr_chunk_causal_attention(const uint16_t* qkv, int32_t d_b, int32_t n_heads,
                                    const int32_t* chunk_end, const int32_t* cu_seqlens_host,
                                    int32_t n_req, int64_t n_tokens, uint16_t* out,
                                    void* stream) {
    if (n_heads < 1 || d_b < 1 || d_b % n_heads != 0 || n_tokens < 1 || n_tokens > INT32_MAX / 2)
        return CR_ERR_INVALID_ARG;
    const int hd = d_b / n_heads;
    if (hd != 32 && hd != 64) return CR_ERR_UNSUPPORTED;
    if (!all_aligned(qkv, chunk_end, out)) return CR_ERR_INVALID_ARG;
    Dims d{};
    d.db = d_b;
    d.nh = n_heads;
    d.hd = hd;
    AttnParams* ap = new AttnParams();
    cr_status s = attn_params(d, CR_MASK_BLOCK_CAUSAL, chunk_end, nullptr, cu_seqlens_host, n_req,
                              n_tokens, out, nullptr, ap);
    if (s == CR_OK) {
        ap->status = device_status_ptr();
        s = ap->status ? launch_attention(qkv, n_tokens, hd, *ap, static_cast<cudaStream_t>(stream))
                       : CR_ERR_CUDA;
    }
    delete ap;
    return s;
}

cr_status cr_masked_attention(const uint16_t* qkv, int32_t d_b, int32_t n_heads,
                              int32_t mask_mode, const int32_t* chunk_end,
                              const int32_t* chunk_start, const int32_t* cu_seqlens_host,
                              int32_t n_req, int64_t n_tokens, uint16_t* out, void* stream) {
    if (n_heads < 1 || d_b < 1 || d_b % n_heads != 0 || n_tokens < 1 || n_tokens > INT32_MAX / 2)
        return CR_ERR_INVALID_ARG;
    const int hd = d_b / n_heads;
    if (hd != 32 && hd != 64) return CR_ERR_UNSUPPORTED;
    if (!all_aligned(qkv, out)) return CR_ERR_INVALID_ARG;
    Dims d{};
    d.db = d_b;
    d.nh = n_heads;
    d.hd = hd;
    AttnParams* ap = new AttnParams();
    cr_status s = attn_params(d, mask_mode, chunk_end, chunk_start, cu_seqlens_host, n_req,
                              n_tokens, out, nullptr, ap);
    if (s == CR_OK) {
        ap->status = device_status_ptr();
        s = ap->status ? launch_attention(qkv, n_tokens, hd, *ap, static_cast<cudaStream_t>(stream))
                       : CR_ERR_CUDA;
    }
    delete ap;
    return s;
}

cr_status cr_chunk_starts(const int32_t* chunk_end, const int32_t* cu_seqlens_host, int32_t n_req,
                          int64_t n_tokens, int32_t* chunk_start, void* stream) {
    if (n_tokens < 1 || n_tokens > INT32_MAX / 2 || !all_aligned(chunk_end, chunk_start))
        return CR_ERR_INVALID_ARG;
    Dims d{};
    d.db = 64;
    d.nh = 1;
    d.hd = 64;
    AttnParams* ap = new AttnParams();
    cr_status s = attn_params(d, CR_MASK_BLOCK_DIAGONAL, chunk_end, chunk_start, cu_seqlens_host,
                              n_req, n_tokens, nullptr, nullptr, ap);
    if (s == CR_OK) s = launch_chunk_starts(chunk_end, *ap, n_tokens, chunk_start,
                                            static_cast<cudaStream_t>(stream));
    delete ap;
    return s;
}

cr_status cr_qkv_rope(const uint16_t* u, const uint16_t* w_qkv, const float* b_qkv,
                      const int32_t* pos, int64_t n_tokens, int32_t d_b, int32_t n_heads,
                      float rope_theta, uint16_t* qkv, void* stream) {
    if (n_heads < 1 || d_b < 128 || d_b % 128 != 0 || d_b % n_heads != 0 || n_tokens < 1 ||
        n_tokens > INT32_MAX / 2 || !(rope_theta > 0.0f))
        return CR_ERR_INVALID_ARG;
    const int hd = d_b / n_heads;
    if (hd != 32 && hd != 64) return CR_ERR_UNSUPPORTED;
    if (!all_aligned(u, w_qkv, pos, qkv) || (b_qkv && !aligned16(b_qkv))) return CR_ERR_INVALID_ARG;
    unsigned* status = device_status_ptr();
    if (!status) return CR_ERR_CUDA;
    GemmParams gq{};
    gq.status = status;
    gq.pos = pos;
    gq.bias = b_qkv;
    gq.out = qkv;
    gq.ldo = 3 * d_b;
    gq.rope_dim = hd;
    gq.rope_cols = 2 * d_b;
    repairer_inv_freq(gq.inv_freq, hd, rope_theta);
    return launch_gemm(u, d_b, w_qkv, n_tokens, 3 * d_b, d_b, EPI_QKV_ROPE, gq, nullptr, 0,
                       static_cast<cudaStream_t>(stream));
}

cr_status cr_segment_project(const cr_target_dims* target, int32_t d_seg, const uint16_t* kv,
                             int64_t n_tokens, const uint16_t* w_seg, const float* b_seg,
                             const float* sigma_stale, uint16_t* y, void* workspace,
                             size_t workspace_bytes, void* stream) {
    cr_status s = check_target(target);
    if (s != CR_OK) return s;
    if (d_seg != 8 && d_seg != 16) return CR_ERR_UNSUPPORTED;
    if (n_tokens < 1 || n_tokens > INT32_MAX / 2) return CR_ERR_INVALID_ARG;
    if (!all_aligned(kv, w_seg, b_seg, sigma_stale, y, workspace)) return CR_ERR_INVALID_ARG;
    const Dims d = dims_of(target, nullptr);
    if (workspace_bytes < static_cast<size_t>(d.S * d_seg * d.dh) * 4) return CR_ERR_INVALID_ARG;
    unsigned* status = device_status_ptr();
    if (!status) return CR_ERR_CUDA;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    uint16_t* wfold = static_cast<uint16_t*>(workspace);
    if ((s = launch_fold_sigma(w_seg, sigma_stale, static_cast<int>(d.S), d_seg,
                               static_cast<int>(d.dh), wfold, st)) != CR_OK)
        return s;
    SegParams sp{};
    sp.M = static_cast<int32_t>(n_tokens);
    sp.S = static_cast<int32_t>(d.S);
    sp.d_seg = d_seg;
    sp.b_seg = b_seg;
    sp.y = y;
    sp.ldy = d.S * d_seg;
    sp.status = status;
    return launch_segproj(kv, d.D, wfold, static_cast<int>(d.dh), sp, st);
}

// ------------------------------------------------------------------ training step
// Flat parameter layout (include/cr.h): the trained tensors in a fixed order,
// each starting at a multiple of 8 elements so that every tensor's fp32 and
// bf16 copies are 16-byte aligned.
static int train_tensor_sizes(const Dims& d, int64_t* sz, int max) {
    const int n = 14 + 12 * static_cast<int>(d.B);
    if (n > max) return -1;
    int k = 0;
    sz[k++] = d.S * d.dseg * d.dh;      // w_seg
    sz[k++] = d.S * d.dseg;             // b_seg
    sz[k++] = d.dc * d.S * d.dseg;      // w_map
    sz[k++] = d.dc;                     // b_map
    sz[k++] = d.dc * d.dmodel;          // w_tok
    sz[k++] = d.dc;                     // b_tok
    sz[k++] = d.db * 2 * d.dc;          // w_fuse
    sz[k++] = d.db;                     // b_fuse
    sz[k++] = d.B * d.db * d.dc;        // w_rein
    sz[k++] = d.B * d.db;               // b_rein
    for (int64_t b = 0; b < d.B; ++b) {
        sz[k++] = d.db;                 // ln1_g
        sz[k++] = d.db;                 // ln1_b
        sz[k++] = 3 * d.db * d.db;      // w_qkv
        sz[k++] = 3 * d.db;             // b_qkv
        sz[k++] = d.db * d.db;          // w_o
        sz[k++] = d.db;                 // b_o
        sz[k++] = d.db;                 // ln2_g
        sz[k++] = d.db;                 // ln2_b
        sz[k++] = d.hid * d.db;         // w_fc1
        sz[k++] = d.hid;                // b_fc1
        sz[k++] = d.db * d.hid;         // w_fc2
        sz[k++] = d.db;                 // b_fc2
    }
    sz[k++] = d.db;                     // lnf_g
    sz[k++] = d.db;                     // lnf_b
    sz[k++] = d.D * d.db;               // w_out
    sz[k++] = d.D;                      // b_out
    return k;
}

static int train_offsets(const Dims& d, int64_t* off, int max) {
    int64_t sz[14 + 12 * 64];
    const int n = train_tensor_sizes(d, sz, 14 + 12 * 64);
    if (n < 0 || n + 1 > max) return -1;
    int64_t o = 0;
    for (int i = 0; i < n; ++i) {
        off[i] = o;
        o += (sz[i] + 7) / 8 * 8;
    }
    off[n] = o;
    return n;
}

cr_status cr_param_layout(const cr_target_dims* target, const cr_repairer_dims* rep, int64_t* offsets,
                          int32_t max_offsets) {
    cr_status s = check_target(target);
    if (s == CR_OK) s = check_repairer(rep);
    if (s != CR_OK) return s;
    if (!offsets) return CR_ERR_INVALID_ARG;
    return train_offsets(dims_of(target, rep), offsets, max_offsets) < 0 ? CR_ERR_INVALID_ARG : CR_OK;
}

namespace {
struct TrainLayout {
    size_t inf, h0, rein, blk, blk_stride, hbuf, yf, rope, dz, rowsq, rowscale, losspart, perreq,
        stats_pad, dh, dxm, du, dtmp, pre, gprod, sig16, dqkv, da, lse, dvec, cstart, dse, dy, colsum, colcnt,
        norm, segw, splitk, total;
    size_t x_in, x_mid, u1, u2, qkv, o, g;   // offsets inside one block's region
};

TrainLayout train_layout(const Dims& d, int64_t n) {
    TrainLayout L{};
    size_t off = 0;
    auto take = [&](size_t bytes) {
        const size_t o = off;
        off += align256(bytes);
        return o;
    };
    const size_t N = static_cast<size_t>(n);
    L.inf = take(ws_layout(d, n).total);
    L.h0 = take(N * d.db * 4);
    L.rein = take(N * (d.B > 0 ? d.B : 1) * d.db * 4);
    // per block: x_in, x_mid (fp32), u1, u2 (bf16), qkv (bf16), o (bf16), g (bf16)
    size_t bo = 0;
    auto btake = [&](size_t bytes) {
        const size_t o = bo;
        bo += align256(bytes);
        return o;
    };
    L.x_in = btake(N * d.db * 4);
    L.x_mid = btake(N * d.db * 4);
    L.u1 = btake(N * d.db * 2);
    L.u2 = btake(N * d.db * 2);
    L.qkv = btake(N * 3 * d.db * 2);
    L.o = btake(N * d.db * 2);
    L.g = btake(N * d.hid * 2);
    L.blk_stride = bo;
    L.blk = take(bo * (d.B > 0 ? d.B : 1));
    L.hbuf = take(N * d.db * 4);
    L.yf = take(N * d.db * 2);
    L.rope = take(N * (d.hd / 2) * 8);
    L.dz = take(N * d.D * 2);
    L.rowsq = take(N * 4);
    L.rowscale = take(N * 4);
    L.losspart = take(N * static_cast<size_t>(2 * (d.D / 128)) * 4);   // r^2 per (row, column tile, group)
    L.perreq = take(kMaxReq * 8);
    L.dh = take(N * d.db * 4);
    L.dxm = take(N * d.db * 4);
    L.du = take(N * d.db * 4);
    const int64_t wide = std::max(std::max(d.hid, 3 * d.db), std::max(2 * d.dc, d.S * d.dseg));
    L.dtmp = take(N * d.hid * 4);
    L.pre = take(N * d.hid * 4);
    L.gprod = take(N * d.db * 4);
    L.sig16 = take(N * wide * 2);
    L.dqkv = take(N * 3 * d.db * 4);
    L.da = take(N * d.db * 4);
    L.lse = take(static_cast<size_t>(d.B > 0 ? d.B : 1) * d.nh * N * 4);   // per block [heads][N]
    L.dvec = take(static_cast<size_t>(d.nh) * N * 4);
    L.cstart = take(N * 4);
    L.dse = take(N * 2 * d.dc * 4);
    L.dy = take(N * d.S * d.dseg * 4);
    L.colsum = take(colsum_scratch_floats(n, std::max(d.D, wide)) * 4);
    L.colcnt = take(colsum_counters(std::max(d.D, wide)) * 4);
    L.norm = take(sqnorm_scratch_doubles() * 8);
    L.segw = take(static_cast<size_t>(d.D) * 128 * 4);   // grouped W_seg gradient blocks
    L.splitk = take(8 * N * d.db * 4);                     // split-K parts of the backward's products
    L.total = off;
    return L;
}
}  // namespace

size_t cr_train_workspace_bytes(const cr_target_dims* target, const cr_repairer_dims* rep,
                                int64_t max_tokens, int64_t max_request_tokens) {
    if (check_target(target) != CR_OK || check_repairer(rep) != CR_OK) return 0;
    if (max_tokens < 1 || max_request_tokens < 1 || max_request_tokens > max_tokens ||
        max_tokens > INT32_MAX / 2)
        return 0;
    return train_layout(dims_of(target, rep), max_tokens).total;
}

cr_status cr_train_step(const cr_target_dims* target, const cr_repairer_dims* rep, float* params,
                        uint16_t* params_bf16, float* adam_m, float* adam_v, float* grads,
                        const float* sigma_stale, const float* sigma_delta, const void* kv_stale,
                        const void* kv_joint, const void* emb, const int32_t* chunk_end,
                        const int32_t* pos, const int32_t* cu_seqlens_host, int32_t n_req,
                        int64_t n_tokens, int32_t mask_mode, const cr_adamw* hp, float* stats_out,
                        void* workspace, size_t workspace_bytes, void* stream) {
    cr_status s = check_target(target);
    if (s == CR_OK) s = check_repairer(rep);
    if (s != CR_OK) return s;
    const Dims d = dims_of(target, rep);
    if (d.f32) return CR_ERR_UNSUPPORTED;
    // the backward's products take whole 64-column boxes of every width
    if (d.dc % 64 != 0 || d.dmodel % 64 != 0 || d.hid % 64 != 0 || (d.S * d.dseg) % 64 != 0)
        return CR_ERR_UNSUPPORTED;
    if (!hp || !cu_seqlens_host || n_req < 1 || n_req > kMaxReq || n_tokens < 1 ||
        n_tokens > INT32_MAX / 2 || !valid_mask_mode(mask_mode))
        return CR_ERR_INVALID_ARG;
    if (!(hp->lr >= 0.0f) || !(hp->beta1 >= 0.0f && hp->beta1 < 1.0f) ||
        !(hp->beta2 >= 0.0f && hp->beta2 < 1.0f) || !(hp->eps > 0.0f) || !(hp->weight_decay >= 0.0f) ||
        !(hp->max_grad_norm > 0.0f) || hp->step < 1)
        return CR_ERR_INVALID_ARG;
    if (!all_aligned(params, params_bf16, adam_m, adam_v, grads, sigma_stale, sigma_delta, kv_stale,
                     kv_joint, emb, chunk_end, pos, stats_out, workspace))
        return CR_ERR_INVALID_ARG;
    if (cu_seqlens_host[0] != 0 || cu_seqlens_host[n_req] != n_tokens) return CR_ERR_INVALID_ARG;
    int64_t nmax = 0;
    for (int r = 0; r < n_req; ++r) {
        const int64_t len = cu_seqlens_host[r + 1] - cu_seqlens_host[r];
        if (len < 1) return CR_ERR_INVALID_ARG;
        nmax = std::max(nmax, len);
    }
    const int64_t N = n_tokens;
    const TrainLayout L = train_layout(d, N);
    if (workspace_bytes < L.total) return CR_ERR_INVALID_ARG;
    int64_t off[14 + 12 * 64 + 1];
    const int nt = train_offsets(d, off, 14 + 12 * 64 + 1);
    if (nt < 0) return CR_ERR_INVALID_ARG;
    const int64_t P = off[nt];
    unsigned* status = device_status_ptr();
    if (!status) return CR_ERR_CUDA;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    const float eps = rep->ln_eps;
    const int64_t B = d.B, db = d.db, dc = d.dc, hid = d.hid, hd = d.hd, D = d.D;

    // tensor k of the flat vector: fp32 master, bf16 copy, gradient
    auto pf = [&](int k) { return params + off[k]; };
    auto pb = [&](int k) { return params_bf16 + off[k]; };
    auto gk = [&](int k) { return grads + off[k]; };
    enum { W_SEG, B_SEG, W_MAP, B_MAP, W_TOK, B_TOK, W_FUSE, B_FUSE, W_REIN, B_REIN, BLK0 };
    enum { LN1G, LN1B, WQKV, BQKV, WO, BO, LN2G, LN2B, WFC1, BFC1, WFC2, BFC2 };
    auto bk = [&](int64_t b, int j) { return BLK0 + static_cast<int>(12 * b) + j; };
    const int LNFG = BLK0 + static_cast<int>(12 * B), LNFB = LNFG + 1, W_OUT = LNFG + 2, B_OUT = LNFG + 3;

    // the forward's weights: matrices from the bf16 copy, vectors from the masters
    std::vector<cr_block_weights> blocks(static_cast<size_t>(std::max<int64_t>(B, 1)));
    for (int64_t b = 0; b < B; ++b) {
        cr_block_weights& k = blocks[static_cast<size_t>(b)];
        k.ln1_g = pf(bk(b, LN1G));
        k.ln1_b = pf(bk(b, LN1B));
        k.w_qkv = pb(bk(b, WQKV));
        k.b_qkv = pf(bk(b, BQKV));
        k.w_o = pb(bk(b, WO));
        k.b_o = pf(bk(b, BO));
        k.ln2_g = pf(bk(b, LN2G));
        k.ln2_b = pf(bk(b, LN2B));
        k.w_fc1 = pb(bk(b, WFC1));
        k.b_fc1 = pf(bk(b, BFC1));
        k.w_fc2 = pb(bk(b, WFC2));
        k.b_fc2 = pf(bk(b, BFC2));
    }
    cr_weights w{};
    w.w_seg = pb(W_SEG);
    w.b_seg = pf(B_SEG);
    w.w_map = pb(W_MAP);
    w.b_map = pf(B_MAP);
    w.w_tok = pb(W_TOK);
    w.b_tok = pf(B_TOK);
    w.w_fuse = pb(W_FUSE);
    w.b_fuse = pf(B_FUSE);
    w.w_rein = pb(W_REIN);
    w.b_rein = pf(B_REIN);
    w.blocks = blocks.data();
    w.lnf_g = pf(LNFG);
    w.lnf_b = pf(LNFB);
    w.w_out = pb(W_OUT);
    w.b_out = pf(B_OUT);
    w.sigma_stale = sigma_stale;
    w.sigma_delta = sigma_delta;

    // ---- workspace
    uint8_t* base = static_cast<uint8_t*>(workspace);
    void* inf = base + L.inf;
    const WsLayout IL = ws_layout(d, N);
    // after compress: y rows [y_hi | y_lo], se rows [s_hi e_hi | s_lo e_lo]; the
    // weight gradients take the hi terms as their bf16 operands
    const uint16_t* y = at<uint16_t>(inf, IL.y);
    const uint16_t* se = at<uint16_t>(inf, IL.se2);
    float* h0 = at<float>(base, L.h0);
    float* rein = at<float>(base, L.rein);
    auto blk = [&](int64_t b, size_t o) { return base + L.blk + static_cast<size_t>(b) * L.blk_stride + o; };
    float* H = at<float>(base, L.hbuf);
    uint16_t* yf = at<uint16_t>(base, L.yf);
    float2* rope = at<float2>(base, L.rope);
    uint16_t* DZ = at<uint16_t>(base, L.dz);
    float* ROWSQ = at<float>(base, L.rowsq);
    double* PERREQ = at<double>(base, L.perreq);
    float* DH = at<float>(base, L.dh);
    float* DXM = at<float>(base, L.dxm);
    float* DU = at<float>(base, L.du);
    float* DTMP = at<float>(base, L.dtmp);
    float* PRE = at<float>(base, L.pre);
    float* GPROD = at<float>(base, L.gprod);
    uint16_t* SIG = at<uint16_t>(base, L.sig16);
    float* DQKV = at<float>(base, L.dqkv);
    float* DA = at<float>(base, L.da);
    float* LSE = at<float>(base, L.lse);
    float* DVEC = at<float>(base, L.dvec);
    int32_t* CSTART = at<int32_t>(base, L.cstart);
    float* DSE = at<float>(base, L.dse);
    float* DY = at<float>(base, L.dy);
    float* CS = at<float>(base, L.colsum);
    unsigned* CCNT = at<unsigned>(base, L.colcnt);
    double* NRM = at<double>(base, L.norm);
    float* SEGW = at<float>(base, L.segw);
    float* SPLITK = at<float>(base, L.splitk);
    const size_t splitk_bytes = 8 * static_cast<size_t>(N) * d.db * 4;

    // ---- forward (Sec. 4.1), keeping what the backward needs
    s = cr_compress_features(target, rep, &w, kv_stale, emb, N, h0, rein, inf, IL.total, stream);
    if (s != CR_OK) return s;
    AttnParams* ap = new AttnParams();
    s = attn_params(d, mask_mode, chunk_end, CSTART, cu_seqlens_host, n_req, N, nullptr, status, ap);
    GemmParams gq{};
    gq.status = status;
    gq.pos = pos;
    gq.rope_dim = static_cast<int32_t>(hd);
    gq.rope_cols = static_cast<int32_t>(2 * db);
    repairer_inv_freq(gq.inv_freq, static_cast<int>(hd), rep->rope_theta);
    if (s == CR_OK && B > 0) s = launch_rope_table(pos, N, static_cast<int>(hd / 2), gq.inv_freq, rope, st);
    // chunk starts, for the attention backward's walk of each key tile's queries
    if (s == CR_OK && B > 0) s = launch_chunk_starts(chunk_end, *ap, N, CSTART, st);
    std::unique_ptr<AttnBwdParams> bp_own(new AttnBwdParams());
    AttnBwdParams* bp = bp_own.get();
    bp->chunk_end = chunk_end;
    bp->chunk_start = CSTART;
    bp->d_b = static_cast<int32_t>(db);
    bp->n_heads = static_cast<int32_t>(d.nh);
    bp->n_req = n_req;
    bp->mask_mode = mask_mode;
    bp->scale_log2 = ap->scale_log2;
    bp->scale = static_cast<float>(1.0 / sqrt(static_cast<double>(hd)));
    bp->status = status;
    for (int r = 0; r < n_req; ++r) {
        bp->req_start[r] = cu_seqlens_host[r];
        bp->tile_prefix[r] = bp->n_items;
        bp->n_items += (cu_seqlens_host[r + 1] - cu_seqlens_host[r] + 127) / 128;
    }
    bp->req_start[n_req] = cu_seqlens_host[n_req];
    bp->tile_prefix[n_req] = bp->n_items;
    gq.rope_table = rope;
    GemmParams gr{};
    gr.status = status;
    for (int64_t b = 0; b < B && s == CR_OK; ++b) {
        const cr_block_weights& k = blocks[static_cast<size_t>(b)];
        float* x_in = reinterpret_cast<float*>(blk(b, L.x_in));
        float* x_mid = reinterpret_cast<float*>(blk(b, L.x_mid));
        uint16_t* u1 = reinterpret_cast<uint16_t*>(blk(b, L.u1));
        uint16_t* u2 = reinterpret_cast<uint16_t*>(blk(b, L.u2));
        uint16_t* qkv = reinterpret_cast<uint16_t*>(blk(b, L.qkv));
        uint16_t* o = reinterpret_cast<uint16_t*>(blk(b, L.o));
        uint16_t* g = reinterpret_cast<uint16_t*>(blk(b, L.g));
        if ((s = launch_layernorm(b == 0 ? h0 : H, rein + b * db, B * db, x_in, k.ln1_g, k.ln1_b, eps, N, db,
                                  u1, st)) != CR_OK)
            break;
        gq.bias = k.b_qkv;
        gq.out = qkv;
        gq.ldo = 3 * db;
        if ((s = launch_gemm(u1, db, k.w_qkv, N, 3 * db, db, EPI_QKV_ROPE, gq, nullptr, 0, st)) != CR_OK) break;
        ap->out = o;
        ap->lse = LSE + b * d.nh * N;
        if ((s = launch_attention(qkv, N, static_cast<int>(hd), *ap, st)) != CR_OK) break;
        if ((s = cuda_check(cudaMemcpyAsync(x_mid, x_in, static_cast<size_t>(N * db) * 4,
                                            cudaMemcpyDeviceToDevice, st))) != CR_OK)
            break;
        gr.bias = k.b_o;
        gr.out = x_mid;
        gr.ldo = db;
        if ((s = launch_gemm(o, db, k.w_o, N, db, db, EPI_ADD_F32, gr, nullptr, 0, st)) != CR_OK) break;
        if ((s = launch_layernorm(x_mid, nullptr, 0, nullptr, k.ln2_g, k.ln2_b, eps, N, db, u2, st)) != CR_OK)
            break;
        gr.bias = k.b_fc1;
        gr.out = g;
        gr.ldo = hid;
        if ((s = launch_gemm(u2, db, k.w_fc1, N, hid, db, EPI_GELU_BF16, gr, nullptr, 0, st)) != CR_OK) break;
        if ((s = cuda_check(cudaMemcpyAsync(H, x_mid, static_cast<size_t>(N * db) * 4,
                                            cudaMemcpyDeviceToDevice, st))) != CR_OK)
            break;
        gr.bias = k.b_fc2;
        gr.out = H;
        gr.ldo = db;
        if ((s = launch_gemm(g, hid, k.w_fc2, N, db, hid, EPI_ADD_F32, gr, nullptr, 0, st)) != CR_OK) break;
    }
    delete ap;
    if (s != CR_OK) return s;
    if (B == 0 && (s = cuda_check(cudaMemcpyAsync(H, h0, static_cast<size_t>(N * db) * 4,
                                                  cudaMemcpyDeviceToDevice, st))) != CR_OK)
        return s;
    if ((s = launch_layernorm(H, nullptr, 0, nullptr, w.lnf_g, w.lnf_b, eps, N, db, yf, st)) != CR_OK) return s;

    // ---- objective (Sec. 4.2): r = z - (joint - stale) / sigma_Delta in the head's
    // epilogue, which writes dz = c r and the rows' r^2 sums
    LossParams* lp = new LossParams();
    lp->n_req = n_req;
    for (int r = 0; r <= n_req; ++r) lp->req_start[r] = cu_seqlens_host[r];
    for (int r = 0; r < n_req; ++r)
        lp->scale[r] = static_cast<float>(
            2.0 / (static_cast<double>(cu_seqlens_host[r + 1] - cu_seqlens_host[r]) * D * n_req));
    // the head writes dz and the loss straight from r, which is never stored
    s = launch_loss_head(yf, w.w_out, w.b_out, sigma_delta, static_cast<const uint16_t*>(kv_stale),
                         static_cast<const uint16_t*>(kv_joint), N, D, db, *lp, DZ,
                         reinterpret_cast<float*>(base + L.rowscale), reinterpret_cast<float*>(base + L.losspart),
                         ROWSQ, stats_out, PERREQ, status, st);
    delete lp;
    if (s != CR_OK) return s;

    // ---- backward: the chain rule in reverse, gradients straight into `grads`
    if ((s = cuda_check(cudaMemsetAsync(grads, 0, static_cast<size_t>(P) * 4, st))) != CR_OK) return s;
    // column-sum election counters start at zero (each use leaves them at zero)
    if ((s = cuda_check(cudaMemsetAsync(CCNT, 0, colsum_counters(std::max(d.D, std::max(std::max(d.hid, 3 * d.db),
                                                                           std::max(2 * d.dc, d.S * d.dseg)))) *
                                                     4,
                                        st))) != CR_OK)
        return s;
    // The backward's products on the tensor cores: C [M, N] fp32 (= or, with acc,
    // +=) op(A) B, B stored [K, N]; op(A) = A [M, K], or A^T for A stored [K, M]
    auto mm = [&](const uint16_t* A, int64_t lda, bool a_trans, const uint16_t* B, int64_t ldb, int64_t M,
                  int64_t Nc, int64_t K, float* C, int64_t ldc, bool acc) {
        GemmParams gp{};
        gp.status = status;
        gp.out = C;
        gp.ldo = ldc;
        return launch_gemm_lay(A, lda, a_trans ? LAY_MM : LAY_KM, B, ldb, M, Nc, K, acc ? EPI_ADD_F32 : EPI_F32,
                               gp, st, SPLITK, splitk_bytes);
    };
    auto colsum = [&](const void* a, bool bf16, int64_t cols, int64_t lda, float* out) {
        return launch_colsum(a, bf16, N, cols, lda, out, false, CS, CCNT, st);
    };
    auto to16 = [&](const float* a, int64_t n, uint16_t* out) { return launch_to_bf16(a, n, out, st); };
    // a bias gradient and the bf16 copy of the same fp32 signal, in one pass
    auto colsum16 = [&](const float* a, int64_t cols, uint16_t* a16, float* out) {
        return launch_colsum_bf16(a, N, cols, a16, out, CS, CCNT, st);
    };
#define CR_TRY(x)                   \
    do {                            \
        if ((s = (x)) != CR_OK) return s; \
    } while (0)
    // head: dW_out = dz^T y_f, db_out = sum_t dz, dy_f = dz W_out
    CR_TRY(mm(DZ, D, true, yf, db, D, db, N, gk(W_OUT), db, false));
    CR_TRY(colsum(DZ, true, D, D, gk(B_OUT)));
    CR_TRY(mm(DZ, D, false, pb(W_OUT), db, N, db, D, DU, db, false));
    CR_TRY(launch_ln_backward(H, w.lnf_g, DU, nullptr, eps, N, static_cast<int>(db), DH, GPROD, st));
    CR_TRY(colsum(GPROD, false, db, db, gk(LNFG)));
    CR_TRY(colsum(DU, false, db, db, gk(LNFB)));
    CR_TRY(cuda_check(cudaMemsetAsync(DSE, 0, static_cast<size_t>(N * 2 * dc) * 4, st)));
    for (int64_t b = B - 1; b >= 0; --b) {
        const float* x_in = reinterpret_cast<const float*>(blk(b, L.x_in));
        const float* x_mid = reinterpret_cast<const float*>(blk(b, L.x_mid));
        const uint16_t* u1 = reinterpret_cast<const uint16_t*>(blk(b, L.u1));
        const uint16_t* u2 = reinterpret_cast<const uint16_t*>(blk(b, L.u2));
        const uint16_t* qkv = reinterpret_cast<const uint16_t*>(blk(b, L.qkv));
        const uint16_t* o = reinterpret_cast<const uint16_t*>(blk(b, L.o));
        const uint16_t* g = reinterpret_cast<const uint16_t*>(blk(b, L.g));
        // h = x_mid + W_fc2 g + b_fc2
        CR_TRY(colsum16(DH, db, SIG, gk(bk(b, BFC2))));
        CR_TRY(mm(SIG, db, true, g, hid, db, hid, N, gk(bk(b, WFC2)), hid, false));
        CR_TRY(mm(SIG, db, false, pb(bk(b, WFC2)), hid, N, hid, db, DTMP, hid, false));
        // g = GELU(pre), pre = W_fc1 u2 + b_fc1 (recomputed in fp32)
        GemmParams gp{};
        gp.status = status;
        gp.bias = pf(bk(b, BFC1));
        gp.out = PRE;
        gp.ldo = hid;
        CR_TRY(launch_gemm(u2, db, pb(bk(b, WFC1)), N, hid, db, EPI_F32, gp, nullptr, 0, st));
        CR_TRY(launch_gelu_backward(DTMP, PRE, N * hid, st));
        CR_TRY(colsum16(DTMP, hid, SIG, gk(bk(b, BFC1))));
        CR_TRY(mm(SIG, hid, true, u2, db, hid, db, N, gk(bk(b, WFC1)), db, false));
        CR_TRY(mm(SIG, hid, false, pb(bk(b, WFC1)), db, N, db, hid, DU, db, false));
        // u2 = LN2(x_mid): dx_mid = dh + LN2 backward
        CR_TRY(launch_ln_backward(x_mid, pf(bk(b, LN2G)), DU, DH, eps, N, static_cast<int>(db), DXM, GPROD, st));
        CR_TRY(colsum(GPROD, false, db, db, gk(bk(b, LN2G))));
        CR_TRY(colsum(DU, false, db, db, gk(bk(b, LN2B))));
        // x_mid = x_in + W_o a + b_o
        CR_TRY(colsum16(DXM, db, SIG, gk(bk(b, BO))));
        CR_TRY(mm(SIG, db, true, o, db, db, db, N, gk(bk(b, WO)), db, false));
        CR_TRY(mm(SIG, db, false, pb(bk(b, WO)), db, N, db, db, DA, db, false));
        // attention: the fused backward (P recomputed from the forward's log-sum-exp,
        // dQ, dK, dV into dqkv), dO in bf16 for its MMAs
        CR_TRY(to16(DA, N * db, SIG));
        bp->lse = LSE + b * d.nh * N;
        bp->dqkv = DQKV;
        CR_TRY(launch_attention_backward(qkv, SIG, DA, o, N, static_cast<int>(hd), *bp, DVEC, st));
        CR_TRY(launch_rope_backward(DQKV, rope, N, static_cast<int>(db), static_cast<int>(hd), st));
        // qkv = W_qkv u1 + b_qkv;  u1 = LN1(x_in): dx_in = dx_mid + LN1 backward
        CR_TRY(colsum16(DQKV, 3 * db, SIG, gk(bk(b, BQKV))));
        CR_TRY(mm(SIG, 3 * db, true, u1, db, 3 * db, db, N, gk(bk(b, WQKV)), db, false));
        CR_TRY(mm(SIG, 3 * db, false, pb(bk(b, WQKV)), db, N, db, 3 * db, DU, db, false));
        CR_TRY(launch_ln_backward(x_in, pf(bk(b, LN1G)), DU, DXM, eps, N, static_cast<int>(db), DH, GPROD, st));
        CR_TRY(colsum(GPROD, false, db, db, gk(bk(b, LN1G))));
        CR_TRY(colsum(DU, false, db, db, gk(bk(b, LN1B))));
        // x_in = h^{b-1} + W_rein,b s + b_rein,b: ds += dx_in W_rein,b
        CR_TRY(colsum16(DH, db, SIG, gk(B_REIN) + b * db));
        CR_TRY(mm(SIG, db, true, se, 4 * dc, db, dc, N, gk(W_REIN) + b * db * dc, dc, false));
        CR_TRY(mm(SIG, db, false, pb(W_REIN) + b * db * dc, dc, N, dc, db, DSE, 2 * dc, true));
    }
    // h0 = W_fuse [s; e] + b_fuse
    CR_TRY(colsum16(DH, db, SIG, gk(B_FUSE)));
    CR_TRY(mm(SIG, db, true, se, 4 * dc, db, 2 * dc, N, gk(W_FUSE), 2 * dc, false));
    CR_TRY(mm(SIG, db, false, pb(W_FUSE), 2 * dc, N, 2 * dc, db, DSE, 2 * dc, true));
    // e = W_tok emb + b_tok;  s = W_map y + b_map
    CR_TRY(to16(DSE, N * 2 * dc, SIG));
    CR_TRY(mm(SIG + dc, 2 * dc, true, static_cast<const uint16_t*>(emb), d.dmodel, dc, d.dmodel, N, gk(W_TOK),
              d.dmodel, false));
    CR_TRY(colsum(DSE + dc, false, dc, 2 * dc, gk(B_TOK)));
    const int64_t Sd = d.S * d.dseg;
    CR_TRY(mm(SIG, 2 * dc, true, y, 2 * Sd, dc, Sd, N, gk(W_MAP), Sd, false));
    CR_TRY(colsum(DSE, false, dc, 2 * dc, gk(B_MAP)));
    CR_TRY(mm(SIG, 2 * dc, false, pb(W_MAP), Sd, N, Sd, dc, DY, Sd, false));
    // y_{t,s} = (W_seg,s / sigma_stale) kv_{t,s} + b_seg,s: per segment kv_s^T dy_s
    // ([d_h, d_seg], summed over tokens), then / sigma_stale.  One grouped product:
    // the d_h rows of 128 / d_seg consecutive segments share one 128-column block
    // of dy, the block holding their own d_seg columns; their other columns are
    // computed and dropped (the product reads kv once, which bounds it).
    CR_TRY(colsum16(DY, Sd, SIG, gk(B_SEG)));
    {
        GemmParams gp{};
        gp.status = status;
        gp.out = SEGW;
        gp.ldo = 128;
        gp.bgroup_rows = static_cast<int32_t>((128 / d.dseg) * d.dh);
        CR_TRY(launch_gemm_lay(static_cast<const uint16_t*>(kv_stale), D, LAY_MM, SIG, Sd, D, 128, N, EPI_F32, gp,
                               st));
    }
    CR_TRY(launch_seg_grad(SEGW, gk(W_SEG), d.S, d.dseg, d.dh, sigma_stale, st));

    // ---- clipping and AdamW (App. A)
    AdamWParams ah{};
    ah.lr = hp->lr;
    ah.b1 = hp->beta1;
    ah.b2 = hp->beta2;
    ah.eps = hp->eps;
    ah.wd = hp->weight_decay;
    ah.bc1 = static_cast<float>(1.0 - pow(static_cast<double>(hp->beta1), hp->step));
    ah.bc2 = static_cast<float>(1.0 - pow(static_cast<double>(hp->beta2), hp->step));
    CR_TRY(launch_clip_adamw(params, adam_m, adam_v, grads, params_bf16, P, ah, hp->max_grad_norm, NRM, stats_out,
                             st));
#undef CR_TRY
    return CR_OK;
}

cr_status cr_wait_selftest(void* stream) {
    unsigned* status = device_status_ptr();
    if (!status) return CR_ERR_CUDA;
    return launch_wait_selftest(status, static_cast<cudaStream_t>(stream));
}

}  // extern "C"
