// cr_segment_project_noalloc: the StaleEncoder stage-1 projection for callers
// that cannot allocate device memory.
//
// Some callers have no way to hand this library a workspace: an inference
// engine plugin whose host code runs under a fixed, pre-planned device memory
// budget, a real-time serving loop that must never call cudaMalloc (it can
// synchronise the device and stall every stream), or code running where the
// allocator is unavailable.  This entry point needs no workspace: its only
// scratch, the weight copy with 1/sigma_stale folded in (two bf16 terms per
// weight), lives in a file-scope device array of fixed size that every GPU
// loading the library holds until the process exits.
#include <mutex>

#include "cr_internal.h"

// Largest weight this entry point accepts: S * d_seg * d_h values (the 8B-shape
// target has 1 Mi).  The folded copy keeps two bf16 terms per value: 8 MiB.
#define CR_NOALLOC_SCRATCH_ELEMS (2u * 1024u * 1024u)

static __device__ __align__(256) uint16_t g_noalloc_scratch[2u * CR_NOALLOC_SCRATCH_ELEMS];

namespace {
std::mutex g_noalloc_mu;
uint16_t* g_noalloc_ptr[64];   // device address of g_noalloc_scratch, per device

// Host code cannot use g_noalloc_scratch's name as a device address: resolve it
// once per device, with that device current.
uint16_t* scratch_for_current_device(cr_status* err) {
    int dev = -1;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) {
        *err = CR_ERR_CUDA;
        return nullptr;
    }
    std::lock_guard<std::mutex> lk(g_noalloc_mu);
    if (!g_noalloc_ptr[dev]) {
        void* p = nullptr;
        if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess || !p) {
            *err = CR_ERR_CUDA;
            return nullptr;
        }
        g_noalloc_ptr[dev] = static_cast<uint16_t*>(p);
    }
    return g_noalloc_ptr[dev];
}
}  // namespace

extern "C" cr_status cr_segment_project_noalloc(const cr_target_dims* target, int32_t d_seg,
                                                const uint16_t* kv, int64_t n_tokens,
                                                const uint16_t* w_seg, const float* b_seg,
                                                const float* sigma_stale, uint16_t* y,
                                                void* stream) {
    using namespace cr;
    cr_status err = check_target(target);
    if (err != CR_OK) return err;
    if (d_seg != 8 && d_seg != 16) return CR_ERR_UNSUPPORTED;
    if (n_tokens < 1 || n_tokens > INT32_MAX / 2) return CR_ERR_INVALID_ARG;
    if (!kv || !w_seg || !b_seg || !sigma_stale || !y) return CR_ERR_INVALID_ARG;
    if (!aligned16(kv) || !aligned16(w_seg) || !aligned16(b_seg) || !aligned16(sigma_stale) ||
        !aligned16(y))
        return CR_ERR_INVALID_ARG;
    // S is bounded before the product so that the size check cannot wrap
    const int64_t S = 2ll * target->n_layers * target->n_kv_heads;
    const int64_t per_seg = static_cast<int64_t>(d_seg) * target->head_dim;
    if (S > static_cast<int64_t>(CR_NOALLOC_SCRATCH_ELEMS) / per_seg) return CR_ERR_UNSUPPORTED;
    uint16_t* scratch = scratch_for_current_device(&err);
    if (!scratch) return err;
    unsigned* status = device_status_ptr();
    if (!status) return CR_ERR_CUDA;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    // Every element the projection reads from the scratch is rewritten here
    // first, so nothing has to be cleared between calls.
    cr_status s = launch_fold_sigma(w_seg, sigma_stale, static_cast<int>(S), d_seg,
                                    target->head_dim, scratch, st);
    if (s != CR_OK) return s;
    SegParams sp{};
    sp.M = static_cast<int32_t>(n_tokens);
    sp.S = static_cast<int32_t>(S);
    sp.d_seg = d_seg;
    sp.b_seg = b_seg;
    sp.y = y;
    sp.ldy = S * d_seg;
    sp.status = status;
    return launch_segproj(kv, S * target->head_dim, scratch, target->head_dim, sp, st);
}
